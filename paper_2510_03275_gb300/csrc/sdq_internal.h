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
int build_tables(const sdq_layer_desc* d, const int8_t* signs, float* a_enc, float* g, double* dt = nullptr);

constexpr int kMaxDecodeM = 64;

// e4m3 terms per activation on the decode path.  Up to N = M T = 32 MMA
// columns the accumulators stay double-buffered and the MMA costs the same,
// so batches up to 8 take four terms (~2^-16 relative); larger ones take two
// (~2^-8, the level of the single bf16 rounding of x_tilde on the prefill
// path).
inline int decode_terms(int M) { return M <= 8 ? 4 : 2; }

// G in the order the decode kernel's B-operand builders load it (only when
// B % 16 == 0 and n_b % 8 == 0): for code tile jt (rows j = 8 jt .. 8 jt + 7),
// k batch kb of kbw = min(64, B) inputs and lane (g, t) of the warp MMA, the
// run of R = kbw / 4 inputs i = kb kbw + t R + e (e < R) of row j = 8 jt + g
// at element 2 R (32 (jt (B / kbw) + kb) + lane), as 32-bit words that
// alternate a hi pair (inputs e, e + 1) and the lo pair of the same inputs.
// Within the batch, input t R + 4 s + r is MMA K index 2t + (r & 1) + 8 (r >> 1)
// of 16-deep step s, so that each lane's fragments are one contiguous run.
#ifdef __CUDACC__
__host__ __device__
#endif
inline int g_frag_batch(int B) { return B < 64 ? B : 64; }

// Polyphase table of D^T for the decode kernel's own activation build.
// With n_b / B = p / q in lowest terms, band-limited resampling commutes with
// a cyclic shift of q inputs (p codes), so row r + p m of D^T is row r
// shifted by q m:  D^T[r + p m][i] = D^T[r][(i - q m) mod B]  (checked at plan
// time), and x_tilde = D^T (Had^T x_b) needs only D^T's first p rows.  Entry
// r * poly_stride(B) + d, d < 2B, holds the pair (D^T[r][d mod B],
// D^T[r][(d + 1) mod B]) as a bf16x2 word (hi) and the pair's bf16
// remainders (lo), so that a run of taps from any start d < B needs no
// wrap-around; after the p * poly_stride(B) entries come B floats
// s_k = d_k / sqrt(B) (1 without the Hadamard transform).  A stride of 8
// (mod 16) entries puts a warp's lookups of two phases in different banks.
#ifdef __CUDACC__
__host__ __device__
#endif
constexpr int poly_stride(int B) { return 2 * B + 8; }
constexpr int kMaxPolyBlock = 256;       // B of the polyphase build (8 inputs per lane)
constexpr int kMaxPolyBytes = 16 * 1024; // table entries, without the B floats

// Launch shape of the decode kernel for one batch size (chosen at plan time).
// Grid = S * P CTAs, one per SM: CTA (s, p) contracts k chunk s (CB blocks
// of 128 codes) against row tiles p, p + P, p + 2P, ...
struct DecodeConfig {
  int M, T, NP;           // batch, e4m3 terms per activation, MMA N (M*T rounded up to 16)
  int S, P, CB;           // k chunks, CTAs per k chunk, 128-code blocks per chunk
  int ring;               // code stages in the shared-memory ring
  int stream;             // 1: each stage's slot also carries its blocks' B operand
                          // rows (no resident per-chunk image; larger batches)
  size_t smem;            // dynamic shared memory of the decode kernel
};

}  // namespace sdq

struct sdq_plan_s {
  sdq_layer_desc desc;
  sdq::Geometry geo;
  int device;
  int sm_count;
  float gnorm;         // max_j sum_k |G[j][k]| (bound of |x_tilde| / max |x|)
  float* d_at;         // encode table, transposed: B x n_b (At[k][j] = A_enc[j][k])
  uint16_t* d_g_hi;    // G as bf16 hi part, n_b x B row-major
  uint16_t* d_g_lo;    // G - hi as bf16, n_b x B row-major
  uint16_t* d_g_frag;  // G hi + lo in warp-fragment order (g_frag_index), or null
  uint32_t* d_poly;    // polyphase table of D^T (poly_stride), or null
  int poly_p, poly_q;  // n_b / B = poly_p / poly_q in lowest terms
  int poly_bytes;      // bytes of the table's entries (the B floats follow)
  sdq::DecodeConfig dcfg[sdq::kMaxDecodeM + 1];  // decode launch shape per batch size
};
