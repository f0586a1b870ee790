// K2: plain <-> tiled code layouts (layout maps in include/sdq.h).
//
// Both layouts keep each row's codes in natural order inside groups of 64
// codes, so the tiled layout is a regrouping of plain-layout runs of wpg
// words (16 bytes ternary, 8 bytes binary): run (row, group G) of the plain
// layout becomes row r = row % 128 of slab (row / 128, G).
#include "common.cuh"

namespace sdq {

namespace {

struct PackParams {
  int n_out, wpr, wpg, ngroups;
  int64_t total;  // words of the output layout
};

// One thread per tiled word.  Rows past n_out and groups past the plain row
// are padding (0).
__global__ void pack_kernel(const uint32_t* __restrict__ plain, uint32_t* __restrict__ tiled,
                            PackParams p) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= p.total) return;
  const int i = (int)(w % p.wpg);
  const int64_t run = w / p.wpg;                 // (slab, r)
  const int r = (int)(run % kTileRows);
  const int64_t slab = run / kTileRows;
  const int G = (int)(slab % p.ngroups);
  const int64_t row = (slab / p.ngroups) * kTileRows + r;
  const int j = G * p.wpg + i;                   // word of the plain row
  tiled[w] = (row < p.n_out && j < p.wpr) ? __ldg(plain + row * p.wpr + j) : 0u;
}

// One thread per plain word.  Ternary pattern 10 is counted and decoded as 0.
__global__ void unpack_kernel(const uint32_t* __restrict__ tiled, uint32_t* __restrict__ plain,
                              uint32_t* bad, PackParams p, int ternary) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= p.total) return;
  const int64_t row = w / p.wpr;
  const int j = (int)(w - row * p.wpr);
  const int G = j / p.wpg, i = j - G * p.wpg;
  const int64_t tw = ((((row / kTileRows) * p.ngroups + G) * kTileRows) + row % kTileRows) * p.wpg + i;
  uint32_t v = __ldg(tiled + tw);
  if (ternary) {
    const uint32_t invalid = (v >> 1) & ~v & 0x55555555u;   // fields holding 10
    if (invalid) {
      if (bad) atomicAdd(bad, (uint32_t)__popc(invalid));
      v &= ~(invalid | (invalid << 1));
    }
  }
  plain[w] = v;
}

}  // namespace

cudaError_t launch_pack(const sdq_plan_s* pl, const uint32_t* plain, uint32_t* tiled, cudaStream_t st) {
  const Geometry& g = pl->geo;
  PackParams p{g.n_out, g.words_per_row, g.wpg, g.ngroups,
               (int64_t)g.ntiles * g.ngroups * kTileRows * g.wpg};
  const int threads = 256;
  const int64_t blocks = (p.total + threads - 1) / threads;
  pack_kernel<<<(unsigned)blocks, threads, 0, st>>>(plain, tiled, p);
  return cudaGetLastError();
}

cudaError_t launch_unpack(const sdq_plan_s* pl, const uint32_t* tiled, uint32_t* plain,
                          uint32_t* bad, cudaStream_t st) {
  const Geometry& g = pl->geo;
  PackParams p{g.n_out, g.words_per_row, g.wpg, g.ngroups, (int64_t)g.n_out * g.words_per_row};
  const int threads = 256;
  const int64_t blocks = (p.total + threads - 1) / threads;
  unpack_kernel<<<(unsigned)blocks, threads, 0, st>>>(tiled, plain, bad, p, g.bits == 2);
  return cudaGetLastError();
}

}  // namespace sdq
