// Internal declarations shared by the host and CUDA translation units of
// libsdq.  Not part of the C ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include "sdq.h"

namespace sdq {

constexpr int kTileRows = 128;    // rows per tile of the tiled code layout
constexpr int kGroupCodes = 64;   // codes per k group of the tiled code layout

// Geometry derived from a validated descriptor.
struct Geometry {
  int32_t n_out, k_in, block, n_b, nblk;  // n_b = B * OSR, nblk = K / B
  int64_t k_eff;                          // nblk * n_b
  int32_t bits;                           // 2 ternary, 1 binary
  int32_t words_per_row;                  // plain layout
  int32_t ntiles;                         // tiles of kTileRows rows (tiled layout)
  int32_t ngroups;                        // k groups of kGroupCodes codes per tile
  int32_t wpg;                            // words per row per k group (4 ternary, 2 binary)
  int64_t k_eff_pad;                      // K_eff rounded up to 128 codes
};

// Returns SDQ_OK and fills `g`, or SDQ_ERR_INVALID_ARG.
int validate(const sdq_layer_desc* d, Geometry* g);

// Host fp64 construction of the tables (see tables.cpp).
//   a_enc: n_b x B row-major, A_enc[j][k] = fp32(sum_k' U[j][k'] Had[k][k'])
//   g:     n_b x B row-major, G[j][k]     = fp32(sum_k' Dt[j][k'] Had[k][k'])
//   dt:    n_b x B row-major, D^T itself in fp64 (optional)
int build_tables(const sdq_layer_desc* d, const int8_t* signs, float* a_enc, float* g, double* dt = nullptr,
                 float* g_gptq = nullptr);

constexpr int kMaxDecodeM = 64;

// e2m1 terms per activation on the decode path.  Each 32-code group of
// x_tilde is scaled by its own power of two (|x_tilde 2^-e| < 4) and split
// into terms whose error falls 8x per term, so T terms carry x_tilde to
// about 2^-3T of the group's maximum: 6 terms (2^-18) up to 4 batch rows,
// where the MMA N = M T stays within 32 columns, 4 (2^-12) up to 16, 3
// (2^-9, the level of the single bf16 rounding of x_tilde on the prefill
// path) above.
// Large batches (M >= kDenseMinM) run sdq_linear_forward as "rebuild the
// weights, then one dense GEMM" (csrc/dense.cu) where the plan allows it.
constexpr int kDenseMinM = 768;
constexpr int kDenseMaxNb = 384;   // G^T hi + lo resident in shared memory

inline int decode_terms(int M) { return M <= 4 ? 6 : (M <= 16 ? 4 : 3); }

// Launch shape of the decode kernel for one batch size (chosen at plan time).
// Grid = S * P CTAs, one per SM (more in waves only where nothing else fits): CTA (s, p) contracts k chunk s (CB blocks
// of 128 codes) against row tiles p, p + P, p + 2P, ...
struct DecodeConfig {
  int M, T, NP;           // batch, e2m1 terms per activation, MMA N (M*T rounded up to 16)
  int S, P, CB;           // k chunks, CTAs per k chunk, 128-code blocks per chunk
  int ring;               // code stages in the shared-memory ring
  int sb;                 // 128-code blocks per stage
  int nbuf;               // accumulators per pipeline
  int npipe;              // MMA pipelines (issuing warps, each with its accumulators)
  int ns;                 // TMEM A slots (4 or 8)
  int brow;               // B image rows per 128-code block pair in shared memory: 8 when
                          // the M T term rows fit in the first 8-row group (the MMA's rows
                          // 8..NP-1 then read whatever follows and land in accumulator
                          // columns nothing reads), else NP
  int bstream;            // 1: each stage's B image rows and scale words stream into its
                          // ring slot beside the codes (no chunk-resident image), so the
                          // k chunk is not bounded by shared memory
  int slot_bytes;         // ring slot: codes, then (bstream) B rows at boff, scales at soff
  int boff, soff;
  int dbase;              // TMEM column of the first accumulator
  int sfa, sfs, ss, sss;  // TMEM columns of the A scales, of TMEM slot 0's B
                          // scales, between two blocks' B scales, and between
                          // two slots' B scales
  size_t smem;            // dynamic shared memory of the decode kernel
};

}  // namespace sdq

struct sdq_plan_s {
  sdq_layer_desc desc;
  sdq::Geometry geo;
  int device;
  int sm_count;
  float* d_at;         // encode table, transposed: B x n_b (At[k][j] = A_enc[j][k])
  float* d_g32;        // G in fp32, n_b x B row-major (GPTQ block reconstruction)
  uint16_t* d_g_hi;    // G as bf16 hi part, n_b x B row-major
  uint16_t* d_g_lo;    // G - hi as bf16, n_b x B row-major
  uint16_t* d_gt_hi;   // G^T as bf16 hi / lo parts, B x n_b, each 64-code chunk in the
  uint16_t* d_gt_lo;   // code expansion's K order (prefill_pos64); null where the dense
                       // large-batch route does not apply (B != 128, n_b not a multiple
                       // of 64 or above kDenseMaxNb)
  sdq::DecodeConfig dcfg[sdq::kMaxDecodeM + 1];  // decode launch shape per batch size
};
