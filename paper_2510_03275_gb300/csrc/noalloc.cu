// Allocation-free variant of sdq_linear_forward for decode batches.
//
// Some callers cannot hand this library a workspace: a plugin living inside
// a host runtime that owns every device allocation through its own pool
// (and forbids cudaMalloc from third-party code), or a serving loop that
// must not allocate device memory once it has started.  For them this file
// keeps the decode scratch (x_tilde and the fp8 B operand of the two-kernel
// route, split-K partials, tickets and the call record) in one file-scope
// device array of kNoAllocScratchBytes per GPU, reserved when the library is
// loaded and held until the process exits.
//
// The array is shared by every call on a device and keeps whatever the last
// call left in it: tickets and the call record carry a scrambled 48-bit tag
// per call, so stale contents do not count (a leftover word matches a call's
// tag with probability 2^-47), and everything else is written before it is
// read.  Two calls that overlap on the GPU (different streams,
// or different host threads) race on the array.
#include <mutex>

#include "common.cuh"

namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)16 << 20;   // 16 MiB per device

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once
// per device, with that device current).
int scratch_for_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDQ_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return SDQ_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return SDQ_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return SDQ_OK;
}

// Checks shared by the entry point and its status query: batch size, the
// plan's device being current, the scratch size; then the array's address.
int noalloc_scratch(sdq_plan p, int32_t M, void** ws) {
  if (!p || M < 1 || M > sdq::kMaxDecodeM) return SDQ_ERR_INVALID_ARG;
  int st = sdq::sdq_check_device(p);
  if (st != SDQ_OK) return st;
  const size_t need = sdq_workspace_bytes(p, M);
  if (need == 0) return SDQ_ERR_INVALID_ARG;
  if (need > kNoAllocScratchBytes) return SDQ_ERR_WORKSPACE;
  return scratch_for_current_device(ws);
}

}  // namespace

extern "C" size_t sdq_noalloc_scratch_bytes(void) { return kNoAllocScratchBytes; }

extern "C" int sdq_linear_forward_noalloc(sdq_plan p, const uint32_t* codes_tiled, const float* alpha,
                                          const uint16_t* x, int32_t M, float* y, void* stream) {
  void* ws = nullptr;
  const int st = noalloc_scratch(p, M, &ws);
  if (st != SDQ_OK) return st;
  return sdq_linear_forward(p, codes_tiled, alpha, x, M, y, ws, kNoAllocScratchBytes, stream);
}

extern "C" int sdq_noalloc_status(sdq_plan p, int32_t M, void* stream) {
  void* ws = nullptr;
  const int st = noalloc_scratch(p, M, &ws);
  if (st != SDQ_OK) return st;
  return sdq::workspace_record_status(p, M, ws, stream);
}
