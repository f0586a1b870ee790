// K2: plain <-> tiled code layouts (layout maps in include/sdq.h).
#include "common.cuh"

namespace sdq {

namespace {

struct PackParams {
  int n_out, wpr, n_chunks, bits;
  int64_t k_eff;
  int64_t total;  // words of the output layout
};

// Row and column of field f of word (tile, q, L) in the tiled layout.
__device__ __forceinline__ void tiled_field_pos(int bits, int64_t tile, int n_chunks, int q, int L,
                                                int f, int* row, int64_t* k) {
  const int64_t G = tile / n_chunks, c = tile - G * n_chunks;
  const int g = L >> 2, t = L & 3;
  if (bits == 2) {
    const int j = 3 - (f & 3), i = f >> 2;
    *row = (int)(16 * G) + g + 8 * (j & 1);
    *k = 128 * c + 32 * q + 16 * (j >> 1) + 4 * t + i;
  } else {
    const int j = 7 - (f & 7), i = f >> 3;
    *row = (int)(16 * G) + g + 8 * (j & 1);
    *k = 256 * c + 64 * q + 32 * (j >> 2) + 16 * ((j >> 1) & 1) + 4 * t + i;
  }
}

__global__ void pack_kernel(const uint32_t* __restrict__ plain, uint32_t* __restrict__ tiled,
                            PackParams p) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= p.total) return;
  const int64_t tile = w >> 7;
  const int within = (int)(w & 127), q = within >> 5, L = within & 31;
  const int nf = 32 / p.bits, per = nf;
  const uint32_t mask = (1u << p.bits) - 1u;
  uint32_t out = 0;
  for (int f = 0; f < nf; ++f) {
    int row;
    int64_t k;
    tiled_field_pos(p.bits, tile, p.n_chunks, q, L, f, &row, &k);
    if (row < p.n_out && k < p.k_eff) {
      const uint32_t src = __ldg(plain + (size_t)row * p.wpr + (k / per));
      out |= ((src >> (p.bits * (int)(k % per))) & mask) << (p.bits * f);
    }
  }
  tiled[w] = out;
}

// Inverse map for unpack: tiled (word, shift) of code (row, k).
__device__ __forceinline__ void tiled_locate(int bits, int row, int64_t k, int n_chunks,
                                             int64_t* word, int* shift) {
  const int G = row >> 4, r = row & 15, g = r & 7, half = r >> 3;
  if (bits == 2) {
    const int64_t c = k >> 7;
    int kk = (int)(k & 127);
    const int q = kk >> 5; kk &= 31;
    const int h = kk >> 4; kk &= 15;
    const int t = kk >> 2, i = kk & 3;
    const int j = 2 * h + half;
    const int f = 4 * i + (3 - j);
    *word = 128 * ((int64_t)G * n_chunks + c) + 32 * q + 4 * g + t;
    *shift = 2 * f;
  } else {
    const int64_t c = k >> 8;
    int kk = (int)(k & 255);
    const int q = kk >> 6; kk &= 63;
    const int u = kk >> 5; kk &= 31;
    const int h = kk >> 4; kk &= 15;
    const int t = kk >> 2, i = kk & 3;
    const int j = 4 * u + 2 * h + half;
    const int f = 8 * i + (7 - j);
    *word = 128 * ((int64_t)G * n_chunks + c) + 32 * q + 4 * g + t;
    *shift = f;
  }
}

__global__ void unpack_kernel(const uint32_t* __restrict__ tiled, uint32_t* __restrict__ plain,
                              uint32_t* bad, PackParams p) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= p.total) return;
  const int row = (int)(w / p.wpr);
  const int64_t wi = w - (int64_t)row * p.wpr;
  const int per = 32 / p.bits;
  const uint32_t mask = (1u << p.bits) - 1u;
  uint32_t out = 0, nbad = 0;
  for (int f = 0; f < per; ++f) {
    const int64_t k = wi * per + f;
    if (k >= p.k_eff) break;
    int64_t tw;
    int sh;
    tiled_locate(p.bits, row, k, p.n_chunks, &tw, &sh);
    uint32_t fld = (__ldg(tiled + tw) >> sh) & mask;
    if (p.bits == 2 && fld == 2u) { ++nbad; fld = 0u; }
    out |= fld << (p.bits * f);
  }
  plain[w] = out;
  if (bad && nbad) atomicAdd(bad, nbad);
}

}  // namespace

cudaError_t launch_pack(const sdq_plan_s* pl, const uint32_t* plain, uint32_t* tiled, cudaStream_t st) {
  const Geometry& g = pl->geo;
  PackParams p{g.n_out, g.words_per_row, g.n_chunks, g.bits, g.k_eff,
               (int64_t)g.ng * g.n_chunks * 128};
  const int threads = 256;
  const int64_t blocks = (p.total + threads - 1) / threads;
  pack_kernel<<<(unsigned)blocks, threads, 0, st>>>(plain, tiled, p);
  return cudaGetLastError();
}

cudaError_t launch_unpack(const sdq_plan_s* pl, const uint32_t* tiled, uint32_t* plain,
                          uint32_t* bad, cudaStream_t st) {
  const Geometry& g = pl->geo;
  PackParams p{g.n_out, g.words_per_row, g.n_chunks, g.bits, g.k_eff,
               (int64_t)g.n_out * g.words_per_row};
  const int threads = 256;
  const int64_t blocks = (p.total + threads - 1) / threads;
  unpack_kernel<<<(unsigned)blocks, threads, 0, st>>>(tiled, plain, bad, p);
  return cudaGetLastError();
}

}  // namespace sdq
