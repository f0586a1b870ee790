// Internal declarations shared by the host and CUDA translation units of
// libsdq.  Not part of the C ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include "sdq.h"

namespace sdq {

// Geometry derived from a validated descriptor.
struct Geometry {
  int32_t n_out, k_in, block, n_b, nblk;  // n_b = B * OSR, nblk = K / B
  int64_t k_eff;                          // nblk * n_b
  int32_t bits;                           // 2 ternary, 1 binary
  int32_t words_per_row;                  // plain layout
  int32_t ng;                             // row groups of 16
  int32_t kc;                             // codes per tile chunk (128 / 256)
  int32_t n_chunks;                       // chunks per row group
  int64_t k_eff_pad;                      // n_chunks * kc
};

// Returns SDQ_OK and fills `g`, or SDQ_ERR_INVALID_ARG.
int validate(const sdq_layer_desc* d, Geometry* g);

// Host fp64 construction of the tables (see tables.cpp).
//   a_enc: n_b x B row-major, A_enc[j][k] = fp32(sum_k' U[j][k'] Had[k][k'])
//   g:     n_b x B row-major, G[j][k]     = fp32(sum_k' Dt[j][k'] Had[k][k'])
int build_tables(const sdq_layer_desc* d, const int8_t* signs, float* a_enc, float* g);

// Decode-path terms per activation (bf16 hi + lo below 17 rows, hi only
// above) and 8-column MMA tiles for batch M.
inline int decode_terms(int M) { return M <= 16 ? 2 : 1; }
inline int decode_ntiles(int M) { return (M * decode_terms(M) + 7) / 8; }

constexpr int kMaxDecodeM = 64;

// Launch shape of the decode kernel for one batch size (chosen at plan time).
struct DecodeConfig {
  int M, T, NT;           // batch, fp8 terms per activation, 8-column MMA tiles
  int S, R;               // k-slices and row ranges (grid = R x S)
  int WK, WR;             // warps along k and along rows (WK * WR = 8)
  int cps;                // chunks per k-slice
  int rgc;                // row groups per row range
  int P;                  // per-row partial maxima written by the prep kernel
  size_t smem;            // dynamic shared memory of the decode kernel
};

}  // namespace sdq

struct sdq_plan_s {
  sdq_layer_desc desc;
  sdq::Geometry geo;
  int device;
  int sm_count;
  float* d_at;         // encode table, transposed: B x n_b (At[k][j] = A_enc[j][k])
  uint16_t* d_g_hi;    // G as bf16 hi part, n_b x B row-major
  uint16_t* d_g_lo;    // G - hi as bf16, n_b x B row-major
  sdq::DecodeConfig dcfg[sdq::kMaxDecodeM + 1];  // decode launch shape per batch size
};
