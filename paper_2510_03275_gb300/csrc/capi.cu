// C ABI of libsdq (declarations and contracts in include/sdq.h).
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <numeric>
#include <vector>

#include "common.cuh"

namespace sdq {

namespace {

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

uint16_t host_bf16(double v) {
  float f = (float)v;
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}
double host_bf16_value(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

int cuda_status(cudaError_t e) { return e == cudaSuccess ? SDQ_OK : SDQ_ERR_CUDA; }

}  // namespace

// The plan's tables live on the device it was created on; kernels launch on
// the current device.  A call made with another device current would read
// the other GPU's memory, so it is refused.
int sdq_check_device(const sdq_plan_s* p) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDQ_ERR_CUDA;
  return dev == p->device ? SDQ_OK : SDQ_ERR_INVALID_ARG;
}

uint64_t next_call_number() {
  static std::atomic<uint64_t> calls{0};
  return ++calls;
}

uint64_t call_tag(uint64_t n) {
  // odd multipliers and xor-shifts are bijections of 47-bit integers
  constexpr uint64_t kMask = (1ull << 47) - 1;
  uint64_t v = n & kMask;
  v = (v * 0x5DEECE66Dull) & kMask;
  v ^= v >> 23;
  v = (v * 0x2545F4914F6Dull) & kMask;
  v ^= v >> 19;
  return v | (1ull << 47);
}

WsLayout workspace_layout(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  WsLayout L{};
  size_t off = 0;
  L.xt = off;
  if (M <= kMaxDecodeM) {
    const DecodeConfig& dc = pl->dcfg[M];
    off = align_up(off + sizeof(float) * (size_t)M * g.k_eff_pad, 256);   // fp32 x_tilde (two-kernel route)
    const size_t kb = (size_t)(g.k_eff_pad / 128);
    L.bimg = off;                                  // B operand image: ceil(KB / 2) x NP x 128 bytes
    off = align_up(off + (kb + 1) / 2 * dc.NP * 128, 256);
    L.sfbw = off;                                  // B scale words: KB x NP x 4 bytes
    off = align_up(off + kb * dc.NP * 4, 256);
    L.part = off;
    off = align_up(off + (dc.S > 1 ? sizeof(float) * (size_t)dc.S * M * g.ntiles * kTileRows : 0), 256);
    L.cnt = off;                                   // one 64-bit ticket per row tile
    off = align_up(off + sizeof(uint64_t) * (size_t)g.ntiles, 256);
    L.err = off;                                   // call record
    off = align_up(off + 2 * sizeof(uint64_t), 256);
  } else {
    off = align_up(off + sizeof(uint16_t) * (size_t)M * g.k_eff_pad, 256);
    L.what = off;                                  // dense route: W', n_out x k_in bf16
    if (dense_route_applies(pl, M)) off = align_up(off + sizeof(uint16_t) * (size_t)g.n_out * g.k_in, 256);
    L.bimg = L.sfbw = L.part = L.cnt = L.err = off;   // call record only
    off = align_up(off + 2 * sizeof(uint64_t), 256);
  }
  L.total = off;
  return L;
}

}  // namespace sdq

using namespace sdq;

extern "C" int sdq_plan_create(const sdq_layer_desc* desc, const int8_t* had_signs, sdq_plan* out) {
  if (!desc || !out) return SDQ_ERR_INVALID_ARG;
  *out = nullptr;
  Geometry g;
  int st = validate(desc, &g);
  if (st != SDQ_OK) return st;
  int dev = 0, major = 0, minor = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDQ_ERR_CUDA;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return SDQ_ERR_CUDA;
  if (major != 10 || minor != 3) return SDQ_ERR_UNSUPPORTED;

  const size_t tab = (size_t)g.n_b * g.block;
  std::vector<float> a_enc(tab), gm(tab), at(tab), g32(tab);
  std::vector<double> dt(tab);
  st = build_tables(desc, had_signs, a_enc.data(), gm.data(), dt.data(), g32.data());
  if (st != SDQ_OK) return st;
  for (int j = 0; j < g.n_b; ++j)
    for (int k = 0; k < g.block; ++k) at[(size_t)k * g.n_b + j] = a_enc[(size_t)j * g.block + k];
  std::vector<uint16_t> ghi(tab), glo(tab);
  for (size_t i = 0; i < tab; ++i) {
    ghi[i] = host_bf16(gm[i]);
    glo[i] = host_bf16((double)gm[i] - host_bf16_value(ghi[i]));
  }
  // G^T for the dense large-batch route: row k (an input of the block), its
  // n_b codes' weights in the order the code expansion presents them to the
  // tensor cores (within each 64-code chunk, logical code kl at position
  // prefill_pos64(kl)); hi and lo parts as for G
  const bool dense_tabs = g.block == 128 && g.n_b % 64 == 0 && g.n_b <= kDenseMaxNb;
  std::vector<uint16_t> gthi, gtlo;
  if (dense_tabs) {
    gthi.resize(tab);
    gtlo.resize(tab);
    const bool ter = desc->quantizer == SDQ_TERNARY;
    for (int k = 0; k < g.block; ++k)
      for (int j = 0; j < g.n_b; ++j) {
        const size_t dst = (size_t)k * g.n_b + (j & ~63) + prefill_pos64(j & 63, ter);
        gthi[dst] = ghi[(size_t)j * g.block + k];
        gtlo[dst] = glo[(size_t)j * g.block + k];
      }
  }

  sdq_plan_s* p = new (std::nothrow) sdq_plan_s();
  if (!p) return SDQ_ERR_ALLOC;
  p->desc = *desc;
  p->geo = g;
  p->device = dev;
  p->sm_count = sms;
  if (cudaMalloc(&p->d_at, sizeof(float) * tab) != cudaSuccess ||
      cudaMalloc(&p->d_g32, sizeof(float) * tab) != cudaSuccess ||
      cudaMalloc(&p->d_g_hi, sizeof(uint16_t) * tab) != cudaSuccess ||
      cudaMalloc(&p->d_g_lo, sizeof(uint16_t) * tab) != cudaSuccess) {
    sdq_plan_destroy(p);
    return SDQ_ERR_ALLOC;
  }
  if (dense_tabs && (cudaMalloc(&p->d_gt_hi, sizeof(uint16_t) * tab) != cudaSuccess ||
                     cudaMalloc(&p->d_gt_lo, sizeof(uint16_t) * tab) != cudaSuccess)) {
    sdq_plan_destroy(p);
    return SDQ_ERR_ALLOC;
  }
  if (dense_tabs && (cudaMemcpy(p->d_gt_hi, gthi.data(), sizeof(uint16_t) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
                     cudaMemcpy(p->d_gt_lo, gtlo.data(), sizeof(uint16_t) * tab, cudaMemcpyHostToDevice) != cudaSuccess)) {
    sdq_plan_destroy(p);
    return SDQ_ERR_CUDA;
  }
  if (cudaMemcpy(p->d_at, at.data(), sizeof(float) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(p->d_g32, g32.data(), sizeof(float) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(p->d_g_hi, ghi.data(), sizeof(uint16_t) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(p->d_g_lo, glo.data(), sizeof(uint16_t) * tab, cudaMemcpyHostToDevice) != cudaSuccess) {
    sdq_plan_destroy(p);
    return SDQ_ERR_CUDA;
  }
  for (int M = 1; M <= kMaxDecodeM; ++M) p->dcfg[M] = decode_config_search(p, M);
  *out = p;
  return SDQ_OK;
}

extern "C" int sdq_plan_destroy(sdq_plan p) {
  if (!p) return SDQ_ERR_INVALID_ARG;
  cudaError_t e = cudaSuccess, e2;
  if (p->d_at && (e2 = cudaFree(p->d_at)) != cudaSuccess) e = e2;
  if (p->d_g32 && (e2 = cudaFree(p->d_g32)) != cudaSuccess) e = e2;
  if (p->d_g_hi && (e2 = cudaFree(p->d_g_hi)) != cudaSuccess) e = e2;
  if (p->d_g_lo && (e2 = cudaFree(p->d_g_lo)) != cudaSuccess) e = e2;
  if (p->d_gt_hi && (e2 = cudaFree(p->d_gt_hi)) != cudaSuccess) e = e2;
  if (p->d_gt_lo && (e2 = cudaFree(p->d_gt_lo)) != cudaSuccess) e = e2;
  delete p;
  return cuda_status(e);
}

extern "C" size_t sdq_workspace_bytes(sdq_plan p, int32_t M) {
  if (!p || M < 1 || M > (1 << 20)) return 0;
  return workspace_layout(p, M).total;
}

extern "C" int sdq_encode_rows(sdq_plan p, const float* W, uint32_t* codes_plain, float* alpha,
                               void* stream) {
  if (!p || !W || !codes_plain || !alpha) return SDQ_ERR_INVALID_ARG;
  if (!aligned16(W) || !aligned16(codes_plain) || !aligned16(alpha)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_encode(p, W, codes_plain, alpha, (cudaStream_t)stream));
}

extern "C" int sdq_pack(sdq_plan p, const uint32_t* plain, uint32_t* tiled, void* stream) {
  if (!p || !plain || !tiled || !aligned16(plain) || !aligned16(tiled)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_pack(p, plain, tiled, (cudaStream_t)stream));
}

extern "C" int sdq_unpack(sdq_plan p, const uint32_t* tiled, uint32_t* plain, uint32_t* bad_count,
                          void* stream) {
  if (!p || !plain || !tiled || !aligned16(plain) || !aligned16(tiled)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_unpack(p, tiled, plain, bad_count, (cudaStream_t)stream));
}

static int check_ws(sdq_plan p, int32_t M, const void* ws, size_t ws_bytes) {
  if (!p || M < 1 || M > 65535) return SDQ_ERR_INVALID_ARG;
  const int dv = sdq_check_device(p);
  if (dv != SDQ_OK) return dv;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u)) return SDQ_ERR_INVALID_ARG;
  if (ws_bytes < workspace_layout(p, M).total) return SDQ_ERR_WORKSPACE;
  return SDQ_OK;
}

extern "C" int sdq_prep_activations(sdq_plan p, const uint16_t* x, int32_t M, void* ws,
                                    size_t ws_bytes, void* stream) {
  int st = check_ws(p, M, ws, ws_bytes);
  if (st != SDQ_OK) return st;
  if (!x || !aligned16(x)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_prep(p, x, M, ws, (cudaStream_t)stream));
}

static int contract(sdq_plan p, const uint32_t* codes_tiled, const float* alpha, int32_t M, float* y,
                    void* ws, size_t ws_bytes, void* stream, int early, int y_mode) {
  int st = check_ws(p, M, ws, ws_bytes);
  if (st != SDQ_OK) return st;
  if (!codes_tiled || !alpha || !y || !aligned16(codes_tiled) || !aligned16(y)) return SDQ_ERR_INVALID_ARG;
  cudaError_t e = M <= kMaxDecodeM
                      ? launch_decode(p, codes_tiled, alpha, M, y, ws, (cudaStream_t)stream, early, y_mode)
                      : launch_prefill(p, codes_tiled, alpha, M, y, ws, (cudaStream_t)stream);
  if (e == cudaErrorNotSupported) return SDQ_ERR_UNSUPPORTED;
  return cuda_status(e);
}

extern "C" int sdq_contract(sdq_plan p, const uint32_t* codes_tiled, const float* alpha, int32_t M,
                            float* y, void* ws, size_t ws_bytes, void* stream) {
  return contract(p, codes_tiled, alpha, M, y, ws, ws_bytes, stream, 0, kYStore);
}

extern "C" int sdq_contract_add(sdq_plan p, const uint32_t* codes_tiled, const float* alpha, int32_t M,
                                float* y, void* ws, size_t ws_bytes, void* stream) {
  if (M > kMaxDecodeM) return p && M >= 1 ? SDQ_ERR_UNSUPPORTED : SDQ_ERR_INVALID_ARG;
  return contract(p, codes_tiled, alpha, M, y, ws, ws_bytes, stream, 0, kYAdd);
}

// The prepare kernel, then the contraction; behind its own prepare kernel the
// decode kernel may start reading the codes before the preceding grid
// finishes: that grid waited for everything before it in the stream, and it
// does not write the codes.
extern "C" int sdq_linear_forward(sdq_plan p, const uint32_t* codes_tiled, const float* alpha,
                                  const uint16_t* x, int32_t M, float* y, void* ws, size_t ws_bytes,
                                  void* stream) {
  // Decode batches: the prepare kernel also clears y, and the decode kernel
  // adds its split-K partial sums into it with float atomics.
  const bool zero_y = p && M >= 1 && M <= kMaxDecodeM && decode_config(p, M).S > 1;
  int st = check_ws(p, M, ws, ws_bytes);
  if (st != SDQ_OK) return st;
  if (!x || !aligned16(x) || !y || !aligned16(y)) return SDQ_ERR_INVALID_ARG;
  if (M > kMaxDecodeM && dense_route_applies(p, M)) {
    // large batches: rebuild the weights, then one dense GEMM
    if (!codes_tiled || !alpha || !aligned16(codes_tiled)) return SDQ_ERR_INVALID_ARG;
    const cudaError_t e = launch_dense_forward(p, codes_tiled, alpha, x, M, y, ws, (cudaStream_t)stream);
    if (e != cudaErrorNotSupported) return cuda_status(e);
  }
  st = cuda_status(launch_prep(p, x, M, ws, (cudaStream_t)stream, zero_y ? y : nullptr));
  if (st != SDQ_OK) return st;
  return contract(p, codes_tiled, alpha, M, y, ws, ws_bytes, stream, 1, zero_y ? kYZeroed : kYStore);
}

extern "C" int sdq_forward_kernels(sdq_plan p, int32_t M, const uint16_t* x) {
  if (!p || !x || M < 1 || M > 65535) return 0;
  return 2;
}

extern "C" int sdq_forward_route(sdq_plan p, int32_t M) {
  if (!p || M < 1 || M > 65535) return 0;
  if (M <= kMaxDecodeM) return 1;
  return dense_route_applies(p, M) ? 3 : 2;
}

extern "C" int sdq_workspace_status(sdq_plan p, int32_t M, const void* ws, void* stream) {
  if (!p || M < 1 || M > 65535 || !ws) return SDQ_ERR_INVALID_ARG;
  return workspace_record_status(p, M, ws, stream);
}

namespace sdq {
int workspace_record_status(const sdq_plan_s* p, int32_t M, const void* ws, void* stream) {
  const WsLayout L = workspace_layout(p, M);
  uint64_t rec[2] = {0, 0};   // last failed call, last call
  cudaError_t e = cudaMemcpyAsync(rec, static_cast<const uint8_t*>(ws) + L.err, sizeof(rec),
                                  cudaMemcpyDeviceToHost, (cudaStream_t)stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return SDQ_ERR_CUDA;
  return rec[1] != 0 && rec[0] == rec[1] ? SDQ_ERR_TIMEOUT : SDQ_OK;
}
}  // namespace sdq

extern "C" int sdq_read_prep(sdq_plan p, int32_t M, const void* ws, float* xt_out, void* stream) {
  if (!p || M < 1 || M > kMaxDecodeM || !ws || !xt_out) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_read_prep(p, M, ws, xt_out, (cudaStream_t)stream));
}

namespace sdq {

namespace {
__global__ void read_prep_kernel(const float* xt, float* out, int M, int64_t k_eff, int64_t kpad) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)M * k_eff) return;
  const int64_t m = i / k_eff, k = i - m * k_eff;
  out[i] = xt[m * kpad + k];
}
}  // namespace

cudaError_t launch_read_prep(const sdq_plan_s* p, int M, const void* ws, float* out, cudaStream_t st) {
  const WsLayout L = workspace_layout(p, M);
  const float* xt = reinterpret_cast<const float*>(static_cast<const uint8_t*>(ws) + L.xt);
  const int64_t n = (int64_t)M * p->geo.k_eff;
  read_prep_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(xt, out, M, p->geo.k_eff, p->geo.k_eff_pad);
  return cudaGetLastError();
}

}  // namespace sdq
