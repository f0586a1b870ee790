// Base-3 storage of ternary codes: 5 trits per byte (1.6 bits per code, the
// closest byte-aligned rate to eq. (14)'s log2(3) = 1.58 bits).
//
// Row r of the base-3 layout starts at byte r * bpr, bpr = ceil(K_eff / 5)
// rounded up to a multiple of 16; code j is trit t = code mod 3 (0, +1 -> 1,
// -1 -> 2) at digit j mod 5 of byte j / 5 (byte = sum_d t_d 3^d <= 242).
// Both kernels move 80 codes per thread: 16 base-3 bytes <-> 5 plain-layout
// words (16 two-bit fields each), with 16-byte loads / stores on the base-3
// side.
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

// One thread per 80 codes of a row: plain words 5 i .. 5 i + 4 -> base-3
// bytes 16 i .. 16 i + 15.  Codes past K_eff (and the invalid pattern 10)
// give trit 0.  gpr = bpr / 16.
__global__ void pack_base3_kernel(const uint32_t* __restrict__ plain, uint8_t* __restrict__ out, Base3Params p) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= p.total) return;
  const int64_t row = t / p.gpr;
  const int i = (int)(t - row * p.gpr);
  uint32_t w[5];
#pragma unroll
  for (int q = 0; q < 5; ++q) {
    const int j = 5 * i + q;
    w[q] = j < p.wpr ? __ldg(plain + row * p.wpr + j) : 0u;
  }
  const int64_t c0 = (int64_t)kCodesPerThread * i;
  uint32_t bytes[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (int b = 0; b < 16; ++b) {
    uint32_t v = 0;
#pragma unroll
    for (int d = 4; d >= 0; --d) {
      const int c = 5 * b + d;
      const uint32_t f = (w[c >> 4] >> (2 * (c & 15))) & 3u;
      const uint32_t tr = (c0 + c < p.k_eff && (f & 1u)) ? (f >> 1) + 1u : 0u;
      v = 3u * v + tr;
    }
    bytes[b >> 2] |= v << (8 * (b & 3));
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
  const int threads = 256;
  const int64_t blocks = (bp.total + threads - 1) / threads;
  pack_base3_kernel<<<(unsigned)blocks, threads, 0, (cudaStream_t)stream>>>(codes_plain, codes_base3, bp);
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
  const int threads = 256;
  const int64_t blocks = (bp.total + threads - 1) / threads;
  unpack_base3_kernel<<<(unsigned)blocks, threads, 0, (cudaStream_t)stream>>>(codes_base3, codes_plain, bad_count,
                                                                              bp);
  return cudaGetLastError() == cudaSuccess ? SDQ_OK : SDQ_ERR_CUDA;
}
