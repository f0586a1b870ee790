// Base-3 storage of ternary codes: 5 trits per byte (1.6 bits per code, the
// closest byte-aligned rate to eq. (14)'s log2(3) = 1.58 bits).
//
// Row r of the base-3 layout starts at byte r * bpr, bpr = ceil(K_eff / 5)
// rounded up to a multiple of 16; code j is trit t = code mod 3 (0, +1 -> 1,
// -1 -> 2) at digit j mod 5 of byte j / 5 (byte = sum_d t_d 3^d <= 242).
// Both kernels move 80 codes per thread: 16 base-3 bytes <-> 5 plain-layout
// words (16 two-bit fields each), with 16-byte loads / stores on the base-3
// side; the pack kernel stages its plain words through shared memory per
// warp (the unpack kernel stores them directly: staging its stores measured
// slower).
#include "common.cuh"

namespace sdq {

namespace {

constexpr int kCodesPerThread = 80;   // 16 bytes x 5 trits = 5 words x 16 fields

struct Base3Params {
  int n_out, wpr, bpr, gpr;   // plain words / base-3 bytes per row, thread groups per row
  int64_t k_eff, total;       // total = n_out * gpr
};

// The plain field of each trit: 0 -> 00, 1 -> 01 (+1), 2 -> 11 (-1).
__device__ __forceinline__ uint32_t trit_field(uint32_t t) { return t == 0 ? 0u : (t == 1 ? 1u : 3u); }

constexpr int kB3Threads = 256;

// A warp's 32 thread groups own 160 plain words: word i of the warp (i =
// 5 lane' + q) belongs to lane' = i / 5.  Moving them through shared memory
// in the order of i makes consecutive lanes touch consecutive words of a row
// (coalesced) instead of words 20 bytes apart.  Each lane finds the row and
// word of its k-th staged word from lane' (whose row and group index it
// reads by shuffle): ok is false past the row's words or the last group.
__device__ __forceinline__ int64_t warp_word_addr(const Base3Params& p, int64_t row, int gi, bool valid, int k,
                                                 bool& ok) {
  const int i = 32 * k + (threadIdx.x & 31);
  const int src = i / 5, q = i - 5 * src;
  const int64_t r = __shfl_sync(0xffffffffu, row, src);
  const int g = __shfl_sync(0xffffffffu, gi, src);
  const bool v = __shfl_sync(0xffffffffu, valid, src);
  const int j = 5 * g + q;
  ok = v && j < p.wpr;
  return r * p.wpr + j;
}

// One thread per 80 codes of a row: plain words 5 i .. 5 i + 4 -> base-3
// bytes 16 i .. 16 i + 15, through a 1024-entry table from a byte's five
// 2-bit fields (10 bits) to its value (the invalid field 10 reads as trit
// 0); fields of codes past K_eff are cleared first.  gpr = bpr / 16.
__global__ void __launch_bounds__(kB3Threads) pack_base3_kernel(const uint32_t* __restrict__ plain,
                                                                uint8_t* __restrict__ out, Base3Params p) {
  __shared__ uint8_t lut[1024];
  __shared__ uint32_t stage[kB3Threads / 32][160];
  for (int v = threadIdx.x; v < 1024; v += blockDim.x) {
    uint32_t b = 0;
    for (int d = 4; d >= 0; --d) {
      const uint32_t f = (v >> (2 * d)) & 3u;
      b = 3u * b + ((f & 1u) ? (f >> 1) + 1u : 0u);
    }
    lut[v] = (uint8_t)b;
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const bool valid = t < p.total;
  const int64_t row = valid ? t / p.gpr : 0;
  const int i = valid ? (int)(t - row * p.gpr) : 0;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    bool ok;
    const int64_t a = warp_word_addr(p, row, i, valid, k, ok);
    stage[warp][32 * k + lane] = ok ? __ldg(plain + a) : 0u;
  }
  __syncthreads();
  if (!valid) return;
  uint32_t w[6];
#pragma unroll
  for (int q = 0; q < 5; ++q) w[q] = stage[warp][5 * lane + q];
  w[5] = 0u;
  const int64_t c0 = (int64_t)kCodesPerThread * i;
  if (c0 + kCodesPerThread > p.k_eff) {
#pragma unroll
    for (int q = 0; q < 5; ++q) {
      const int64_t keep = p.k_eff - (c0 + 16 * q);
      if (keep <= 0) w[q] = 0u;
      else if (keep < 16) w[q] &= (1u << (2 * keep)) - 1u;
    }
  }
  uint32_t bytes[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (int b = 0; b < 16; ++b) {
    const int bit = 10 * b, q = bit >> 5, sh = bit & 31;
    const uint32_t v = (sh <= 22 ? (w[q] >> sh) : __funnelshift_r(w[q], w[q + 1], sh)) & 0x3FFu;
    bytes[b >> 2] |= (uint32_t)lut[v] << (8 * (b & 3));
  }
  *reinterpret_cast<uint4*>(out + row * p.bpr + 16 * i) = make_uint4(bytes[0], bytes[1], bytes[2], bytes[3]);
}

// One thread per 5 plain words of a row (gpr = ceil(wpr / 5)): base-3 bytes
// 16 i .. 16 i + 15 (0 past bpr) -> plain words 5 i .. 5 i + 4 (those below
// wpr).  Bytes above 242 are counted into *bad and read as five 0 codes;
// codes past K_eff are written as 0 (the plain layout's padding).
__global__ void unpack_base3_kernel(const uint8_t* __restrict__ in, uint32_t* __restrict__ plain, uint32_t* bad,
                                    Base3Params p) {
  __shared__ uint16_t lut[256];   // byte -> its 5 fields (10 bits); 0 for invalid bytes
  for (int v = threadIdx.x; v < 256; v += blockDim.x) {
    uint32_t f = 0, x = (uint32_t)v;
    if (v < 243)
      for (int d = 0; d < 5; ++d) {
        f |= trit_field(x % 3u) << (2 * d);
        x /= 3u;
      }
    lut[v] = (uint16_t)f;
  }
  __syncthreads();
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= p.total) return;
  const int64_t row = t / p.gpr;
  const int i = (int)(t - row * p.gpr);
  uint4 raw = make_uint4(0u, 0u, 0u, 0u);
  if (16 * i < p.bpr) raw = __ldg(reinterpret_cast<const uint4*>(in + row * p.bpr + 16 * i));
  const uint32_t rw[4] = {raw.x, raw.y, raw.z, raw.w};
  uint32_t w[5] = {0u, 0u, 0u, 0u, 0u};
  int nbad = 0;
#pragma unroll
  for (int b = 0; b < 16; ++b) {
    const uint32_t v = (rw[b >> 2] >> (8 * (b & 3))) & 0xFFu;
    nbad += v > 242u;
    const uint32_t f = lut[v];
    const int c = 5 * b;                 // first of the byte's codes; 10 bits from field c
    const int q = c >> 4, s = 2 * (c & 15);
    w[q] |= f << s;
    if (s > 22) w[q + 1] |= f >> (32 - s);
  }
  if (nbad && bad) atomicAdd(bad, (uint32_t)nbad);
  const int64_t c0 = (int64_t)kCodesPerThread * i;
#pragma unroll
  for (int q = 0; q < 5; ++q) {
    const int j = 5 * i + q;
    if (j >= p.wpr) break;
    // keep the fields of codes below K_eff
    const int64_t first = c0 + 16 * q;
    const int64_t keep = p.k_eff - first;
    uint32_t v = w[q];
    if (keep <= 0) v = 0u;
    else if (keep < 16) v &= (1u << (2 * keep)) - 1u;
    plain[row * p.wpr + j] = v;
  }
}

int base3_bytes_per_row(int64_t k_eff) { return (int)(16 * (((k_eff + 4) / 5 + 15) / 16)); }

}  // namespace

}  // namespace sdq

using namespace sdq;

extern "C" size_t sdq_base3_bytes(const sdq_layer_desc* desc) {
  Geometry g;
  if (validate(desc, &g) != SDQ_OK || desc->quantizer != SDQ_TERNARY) return 0;
  return (size_t)g.n_out * base3_bytes_per_row(g.k_eff);
}

extern "C" int sdq_pack_base3(sdq_plan p, const uint32_t* codes_plain, uint8_t* codes_base3, void* stream) {
  if (!p || !codes_plain || !codes_base3) return SDQ_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(codes_plain) | reinterpret_cast<uintptr_t>(codes_base3)) & 15u)
    return SDQ_ERR_INVALID_ARG;
  if (p->desc.quantizer != SDQ_TERNARY) return SDQ_ERR_UNSUPPORTED;
  const int dv = sdq_check_device(p);
  if (dv != SDQ_OK) return dv;
  const Geometry& g = p->geo;
  Base3Params bp;
  bp.n_out = g.n_out; bp.wpr = g.words_per_row; bp.bpr = base3_bytes_per_row(g.k_eff);
  bp.gpr = bp.bpr / 16; bp.k_eff = g.k_eff; bp.total = (int64_t)g.n_out * bp.gpr;
  const int64_t blocks = (bp.total + kB3Threads - 1) / kB3Threads;
  pack_base3_kernel<<<(unsigned)blocks, kB3Threads, 0, (cudaStream_t)stream>>>(codes_plain, codes_base3, bp);
  return cudaGetLastError() == cudaSuccess ? SDQ_OK : SDQ_ERR_CUDA;
}

extern "C" int sdq_unpack_base3(sdq_plan p, const uint8_t* codes_base3, uint32_t* codes_plain, uint32_t* bad_count,
                                void* stream) {
  if (!p || !codes_plain || !codes_base3) return SDQ_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(codes_plain) | reinterpret_cast<uintptr_t>(codes_base3)) & 15u)
    return SDQ_ERR_INVALID_ARG;
  if (p->desc.quantizer != SDQ_TERNARY) return SDQ_ERR_UNSUPPORTED;
  const int dv = sdq_check_device(p);
  if (dv != SDQ_OK) return dv;
  const Geometry& g = p->geo;
  Base3Params bp;
  bp.n_out = g.n_out; bp.wpr = g.words_per_row; bp.bpr = base3_bytes_per_row(g.k_eff);
  bp.gpr = (g.words_per_row + 4) / 5; bp.k_eff = g.k_eff; bp.total = (int64_t)g.n_out * bp.gpr;
  const int64_t blocks = (bp.total + kB3Threads - 1) / kB3Threads;
  unpack_base3_kernel<<<(unsigned)blocks, kB3Threads, 0, (cudaStream_t)stream>>>(codes_base3, codes_plain,
                                                                                  bad_count, bp);
  return cudaGetLastError() == cudaSuccess ? SDQ_OK : SDQ_ERR_CUDA;
}
