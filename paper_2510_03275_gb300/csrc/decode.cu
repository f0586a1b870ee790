// K4: decode contraction (M <= 64) on the 5th-generation tensor cores, with
// the code operand expanded into tensor memory.
//
//   y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]        (section 3.5, eq. 12)
//
// A skinny contraction whose cost is streaming the packed codes (2 or 1 bits
// per weight sample) from HBM.  Expanding codes into multiply-accumulate
// operands on the CUDA cores costs more integer issue slots than the HBM rate
// leaves, so the products run on tcgen05.mma kind::f8f6f4 (M = 128, N = NP,
// K = 32 per instruction) and the CUDA cores only expand:
//   A (TMEM)  the codes of a 128-row tile as e4m3 +-2.0 / 0: thread = TMEM
//             lane = weight row, 4 codes per 32-bit column, written with
//             tcgen05.st straight from the shift-and-mask expansion of the
//             row's packed words (no shared-memory round trip)
//   B (smem)  the activations as T e4m3 terms per batch row m:
//             x_tilde[m] * 2^-e_m = sum_t 16^-t q_t[m] (e_m from a bound on |x_tilde[m]|),
//             N = M*T rows rounded up to 16, K-major, 128-byte swizzle:
//             either written for all of K by the decode prepare kernel and
//             then copied by each CTA, the part of its k chunk at once
//             (resident) or each stage's blocks with the stage's codes
//             (streamed, larger batches: decode_kernel<true>), or (small
//             batches, `fused`) built by the CTA's expander warps for its k
//             chunk from x itself, with a scale 2^e_m of its own
//             (build_b_operand)
//   D (TMEM)  fp32, 128 lanes x NP columns
// so that y[m, r] = alpha_r / 2 * 2^e_m * sum_t 16^-t D[r, m T + t].
//
// A stage is up to sb blocks of 128 codes (4 sb MMAs): every mbarrier wait
// of an MMA-issuing thread costs about as much as several MMAs, and one
// thread issues at most one MMA every ~45 cycles, so the CTA runs two
// independent pipelines e = 0, 1 on alternate stages (i = e mod 2), each with
// its own producer thread, two expander sets, MMA issuer, two TMEM slots
// and accumulator; the epilogue adds the two accumulators.  Set t of
// pipeline e owns TMEM slot 2e + t and expands the pipeline's stages
// j = t (mod 2): every mbarrier has one producer and one consumer that both
// walk its phases in order.
//
// CTA (k chunk s, row set p) of one SM, 24 warps:
//   warps 0, 1    lane 0 of warp e streams pipeline e's stages (one 128-row
//                 tile x up to sb * 128 codes = contiguous slabs of the tiled
//                 layout, plus their B rows when streamed) into its
//                 shared-memory ring slots with bulk copies; warp 0 also owns
//                 the TMEM allocation and copies a resident B operand
//   warps 2, 3    lane 0 of warp 2 + e issues pipeline e's MMAs, commits to
//                 the stage's TMEM slot and, after its last stage of a row
//                 tile, to its accumulator
//   warps 4..19   expanders: set x = 2e + t (warps 4 + 4x .. 7 + 4x, one per
//                 TMEM lane quadrant) expands stages i = e + 2t (mod 4) into
//                 TMEM slot x
//   warps 20..23  epilogue: read and add the accumulators, combine the
//                 terms, scale and store y, or store a split-K partial, fence
//                 it and take the tile's ticket while the next tile's MMAs
//                 run; the CTA with the last ticket of a tile sums its S
//                 partials in a fixed order (deterministic)
// With `early` set the producers start the code stream before waiting for
// the preceding grid (codes are never written by the prep kernels).
// Every mbarrier wait is bounded (about 2 s); a timeout writes the call
// number into the workspace's call record and the CTA drains its copies and
// MMAs before freeing TMEM.
#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBlk = 128;                        // codes per block (4 MMAs of K = 32)
constexpr int kProducers = 2;                    // warps 0, 1
constexpr int kIssuerWarp0 = 2;                  // warps 2, 3
constexpr int kSlots = 2;                        // TMEM A slots (and expander sets) per pipeline
constexpr int kMaxSb = 3;                        // at most 3 blocks per stage
constexpr int kExpWarp0 = 4;                     // warps 4..19
constexpr int kExpSets = 2 * kSlots;
constexpr int kEpiWarp0 = kExpWarp0 + 4 * kExpSets;   // warps 20..23
constexpr int kThreads = 32 * (kEpiWarp0 + 4);   // 768
constexpr int kMaxRing = 24;
constexpr int kMaxSpu = 128;                     // stages per row tile (config search bound)
constexpr int kSmemMax = 224 * 1024;
constexpr int kSmemMin = 120 * 1024;             // > half an SM: one CTA per SM
constexpr int kMaxFuseM = 4;                     // batch rows of the fused B operand
constexpr int kBuildThreads = 32 * 4 * kExpSets; // the expander warps build it
constexpr int kMaxBuildSteps = 64;               // 16-deep MMA steps per warp (fusion bound)
constexpr int kFusePre = 4;                      // code stages requested before the B operand is built
constexpr int kRedWords = 64;                    // split-K sums summed CTA-wide: first 2048 tiles
static_assert(kMaxRing <= 32 && 2 * kSlots + 7 <= 16 && kRedWords == 64 && kMaxSpu < 160,
              "the prologue's per-warp set-up assumes these bounds");

struct DecodeParams {
  const uint32_t* codes;
  const float* alpha;
  const uint8_t* bimg;   // B operand image: KB x NP x 128 bytes (prepared path)
  const int* sexp;       // per-batch-row scale exponents e_m (prepared path)
  float* y;              // M x n_out
  float* part;           // S x M x (ntiles * 128) split-K partials
  uint64_t* cnt;         // ntiles split-K tickets (ticket_take)
  uint64_t* rec;         // call record
  uint64_t call;
  // Fused path (fused = 1): the B operand is built in the kernel from x.
  const uint16_t* x;     // M x K bf16 bits
  const uint16_t* g_frag; // G = D^T Had^T, bf16 hi + lo, warp-fragment order (g_frag_batch)
  const uint32_t* poly;  // polyphase table of D^T (poly_stride), then B floats d_k / sqrt(B)
  float gnorm;           // max_j sum_i |G[j, i]| (with margin)
  int fused, K, B, n_b;
  int use_poly, poly_p, poly_q, poly_bytes, fwht;
  int64_t k_eff;
  int M, T, NP, S, P, CB, KB, ring, sb, nbuf, dbase;
  int n_out, ntiles, ngroups, ternary, early, stream;
  uint32_t blk_bytes, slot_bytes, b_bytes;   // b_bytes: resident image (0 when streamed)
};

// Bounded wait whose outcome is the same for all lanes of the warp (the
// tcgen05 loads and stores that follow are warp-collective).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity));
}
// Barrier over `nthreads` threads that also ANDs a predicate across them.
__device__ __forceinline__ bool group_and(int id, int nthreads, bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, %2, %3, p;\n"
      " selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r) : "r"((uint32_t)v), "r"(id), "r"(nthreads) : "memory");
  return r != 0;
}

// Stage j of a row tile (spu stages over the chunk's ncb blocks) covers
// blocks [first, last).
__device__ __forceinline__ int stage_block(int j, int ncb, int spu) { return j * ncb / spu; }

__device__ __forceinline__ float bf16_mag(uint32_t h) { return __uint_as_float((h & 0x7FFFu) << 16); }

// Fused B operand (small decode batches): the expander warps compute x_tilde
// for this CTA's k chunk only,
//   x_tilde[m, b n_b + j] = sum_i G[j, i] x[m, b B + i]      (G = D^T Had^T)
// on warp MMAs with fp32 accumulation, and writes its T e4m3 terms into the
// shared-memory B image, laid out as the decode prepare kernel lays out the
// global one.  The term scale 2^e_m is this CTA's own, from the bound
// |x_tilde[m, k]| <= gnorm max |x[m, i]| over the input blocks the chunk
// reads; the epilogue applies it to this CTA's products only, so no CTA
// waits for another.  Two ways to the same x_tilde:
//   polyphase (B <= 256, use_poly): u = Had^T x_b by a fast Walsh-Hadamard
//     transform, then x_tilde = D^T u with D^T's entries looked up in its
//     polyphase table (a few KB in shared memory); u and D^T as bf16 hi + lo
//   dense: G x_b with bf16 x exact and G as bf16 hi + lo, G's fragments
//     streamed from the plan's fragment-ordered copy (n_b B 4 bytes)
//
// MMA tiles are 16 (m, b) rows x 8 codes j.  Per k batch of kbw inputs each
// lane takes one contiguous run of the inputs (x or u) per row and of the
// matching G or D^T entries: input t R + 4 s + r of the batch is MMA K index
// 2t + (r & 1) + 8 (r >> 1) of step s, for both operands, which leaves the
// dot products unchanged.
struct BuildGeo {
  int64_t k0, k1, kend;   // chunk codes [k0, kend), with a value below k1
  int blo, nbi, rows;     // first input block, input blocks, (m, b) rows (m-major)
  int kbw, R, nkb, S4;    // k batch, run length, batches, 16-deep steps per batch
};

// G fragments of code tile jt, batch kb.
__device__ __forceinline__ void load_g_frags(const DecodeParams& p, const BuildGeo& q, int jt, int kb, int lane,
                                             uint32_t (&gw)[16]) {
  const uint4* gf = reinterpret_cast<const uint4*>(p.g_frag) +
                    ((size_t)(jt * q.nkb + kb) * 32 + lane) * (q.kbw / 16);
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    uint4 v = make_uint4(0, 0, 0, 0);
    if (c < q.kbw / 16) v = __ldg(gf + c);
    gw[4 * c] = v.x; gw[4 * c + 1] = v.y; gw[4 * c + 2] = v.z; gw[4 * c + 3] = v.w;
  }
}

// x runs of rows xa0 / xa1 (lane offset applied) for batch kb.
__device__ __forceinline__ void load_x_frags(const BuildGeo& q, const uint16_t* xa0, const uint16_t* xa1, int kb,
                                             uint32_t (&xw)[2][8]) {
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const bool in = c < q.kbw / 32 || (c == 0 && q.kbw == 16);
    uint4 v0 = make_uint4(0, 0, 0, 0), v1 = v0;
    if (in && q.kbw >= 32) {
      v0 = __ldg(reinterpret_cast<const uint4*>(xa0 + kb * q.kbw) + c);
      v1 = __ldg(reinterpret_cast<const uint4*>(xa1 + kb * q.kbw) + c);
    } else if (in) {   // kbw = 16: R = 4 inputs, 8 bytes per row
      const uint2 h0 = __ldg(reinterpret_cast<const uint2*>(xa0 + kb * q.kbw));
      const uint2 h1 = __ldg(reinterpret_cast<const uint2*>(xa1 + kb * q.kbw));
      v0.x = h0.x; v0.y = h0.y; v1.x = h1.x; v1.y = h1.y;
    }
    xw[0][4 * c] = v0.x; xw[0][4 * c + 1] = v0.y; xw[0][4 * c + 2] = v0.z; xw[0][4 * c + 3] = v0.w;
    xw[1][4 * c] = v1.x; xw[1][4 * c + 1] = v1.y; xw[1][4 * c + 2] = v1.z; xw[1][4 * c + 3] = v1.w;
  }
}

// Separate accumulators for the hi and lo parts of G halve the MMA
// dependency chains; they are summed once per tile.
__device__ __forceinline__ void mma_batch(const BuildGeo& q, const uint32_t (&xw)[2][8], const uint32_t (&gw)[16],
                                          float (&acc)[2][4]) {
#pragma unroll
  for (int s = 0; s < 4; ++s)
    if (s < q.S4) {
      const uint32_t a[4] = {xw[0][2 * s], xw[1][2 * s], xw[0][2 * s + 1], xw[1][2 * s + 1]};
      mma_bf16_16816(acc[0], a, gw[4 * s], gw[4 * s + 2]);       // G words alternate hi and lo pairs
      mma_bf16_16816(acc[1], a, gw[4 * s + 1], gw[4 * s + 3]);
    }
}
__device__ __forceinline__ void acc_sum(const float (&a)[2][4], float (&out)[4]) {
#pragma unroll
  for (int e = 0; e < 4; ++e) out[e] = a[0][e] + a[1][e];
}
// Row stride (floats) of the fp32 x_tilde scratch per (m, 128-code block):
// 128 MMA positions + 4 of padding, so that lanes on different blocks hit
// different banks.
constexpr int kXtStride = 132;

// The lane's four x_tilde values of tile (rows r0, r1; codes 8 jt ..) into
// the scratch, at their MMA position: xs[(m ncb + block) kXtStride + kap].
__device__ __forceinline__ void store_xt(const DecodeParams& p, const BuildGeo& q, float* xs, int ncb, int jt,
                                         int t, int r0, int r1, int m0, int m1, const float (&acc)[4]) {
  const bool ter = p.ternary != 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int rho = e < 2 ? r0 : r1;
    if (rho >= q.rows) continue;
    const int m = e < 2 ? m0 : m1;
    const int64_t k = (int64_t)(q.blo + rho - m * q.nbi) * p.n_b + jt * 8 + 2 * t + (e & 1);
    if (k < q.k0 || k >= q.k1) continue;
    const int kl = (int)(k - q.k0);
    xs[(m * ncb + (kl >> 7)) * kXtStride + decode_pos(kl & 127, ter)] = acc[e];
  }
}

// T e4m3 terms of W = 16 or 8 consecutive MMA positions (all or half of one
// 16-byte chunk of each term row), packed and stored W bytes at a time.
// Position 16 c + h W + i of block blk, batch row m.
template <int T, int W>
__device__ __forceinline__ void chunk_terms(const DecodeParams& p, uint8_t* bop, const float* xs, int ncb, int m,
                                            int blk, int c, int h, float inv, int lim) {
  const bool ter = p.ternary != 0;
  const float4* src = reinterpret_cast<const float4*>(xs + (m * ncb + blk) * kXtStride + 16 * c + W * h);
  float v[W];
#pragma unroll
  for (int i = 0; i < W / 4; ++i) {
    const float4 f = src[i];
    v[4 * i] = f.x; v[4 * i + 1] = f.y; v[4 * i + 2] = f.z; v[4 * i + 3] = f.w;
  }
#pragma unroll
  for (int i = 0; i < W; ++i)   // padding codes (k >= K_eff) are 0; the scratch is not written there
    v[i] = blk * kBlk + decode_stage_k(16 * c + W * h + i, ter) < lim ? v[i] * inv : 0.f;
  uint8_t* base = bop + (size_t)blk * p.NP * 128;
#pragma unroll
  for (int tt = 0; tt < T; ++tt) {
    uint32_t w[W / 4];
#pragma unroll
    for (int i = 0; i < W / 4; ++i) {
      uint32_t b4 = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t qb = f32_to_e4m3(v[4 * i + j]);
        b4 |= qb << (8 * j);
        if (tt + 1 < T) v[4 * i + j] = (v[4 * i + j] - e4m3_to_f32(qb)) * 16.f;
      }
      w[i] = b4;
    }
    const int row = m * T + tt;
    uint8_t* dst = base + row * 128 + ((c ^ (row & 7)) << 4) + W * h;
    if constexpr (W == 16)
      *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
    else
      *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
  }
}

template <int W>
__device__ __forceinline__ void all_terms(const DecodeParams& p, uint8_t* bop, const float* xs, int ncb, int et,
                                          const float* inv_s, int lim) {
  constexpr int PER = 128 / W;   // tasks per (m, block)
  for (int task = et; task < p.M * ncb * PER; task += kBuildThreads) {
    const int m = task / (ncb * PER), rem = task - m * ncb * PER, blk = rem / PER, cw = rem % PER;
    const int c = cw / (16 / W), h = cw % (16 / W);
    const float inv = inv_s[m];
    switch (p.T) {
      case 4: chunk_terms<4, W>(p, bop, xs, ncb, m, blk, c, h, inv, lim); break;
      case 3: chunk_terms<3, W>(p, bop, xs, ncb, m, blk, c, h, inv, lim); break;
      default: chunk_terms<2, W>(p, bop, xs, ncb, m, blk, c, h, inv, lim); break;
    }
  }
}

// Polyphase build: u = Had^T x_b of one (m, b) row, V = B / 32 inputs per
// lane (lanes beyond B / V idle), by a fast Walsh-Hadamard transform with
// the sign and 1 / sqrt(B) scale applied first; stored as bf16 hi + lo rows
// of stride us; returns the lane's max |x|.
template <int V>
__device__ __forceinline__ float row_transform(const DecodeParams& p, const uint16_t* xr, bool act, int lane,
                                               uint16_t* uhi, uint16_t* ulo) {
  float v[V];
  uint32_t w[(V + 1) / 2];
#pragma unroll
  for (int i = 0; i < (V + 1) / 2; ++i) w[i] = 0u;
  if (act) {
    if constexpr (V == 8) {
      const uint4 t4 = __ldg(reinterpret_cast<const uint4*>(xr));
      w[0] = t4.x; w[1] = t4.y; w[2] = t4.z; w[3] = t4.w;
    } else if constexpr (V == 4) {
      const uint2 t2 = __ldg(reinterpret_cast<const uint2*>(xr));
      w[0] = t2.x; w[1] = t2.y;
    } else if constexpr (V == 2) {
      w[0] = __ldg(reinterpret_cast<const uint32_t*>(xr));
    } else {
      w[0] = __ldg(reinterpret_cast<const unsigned short*>(xr));
    }
  }
  float mx = 0.f;
#pragma unroll
  for (int e = 0; e < V; ++e) {
    v[e] = __uint_as_float((e & 1) ? (w[e >> 1] & 0xFFFF0000u) : (w[e >> 1] << 16));
    mx = fmaxf(mx, fabsf(v[e]));
  }
  if (act) {
    const float* sg = reinterpret_cast<const float*>(p.poly) + p.poly_bytes / 4 + lane * V;
#pragma unroll
    for (int e = 0; e < V; ++e) v[e] *= __ldg(sg + e);
  }
  if (p.fwht) {
#pragma unroll
    for (int h = 1; h < V; h <<= 1)   // butterflies within the lane
#pragma unroll
      for (int e = 0; e < V; ++e)
        if (!(e & h)) {
          const float a = v[e], b = v[e + h];
          v[e] = a + b;
          v[e + h] = a - b;
        }
    for (int o = 1; o < p.B / V; o <<= 1)   // across lanes: index bit o * V
#pragma unroll
      for (int e = 0; e < V; ++e) {
        const float other = __shfl_xor_sync(0xffffffffu, v[e], o);
        v[e] = (lane & o) ? other - v[e] : v[e] + other;
      }
  }
  if (lane * V < p.B) {
    uint16_t hb[V], lb[V];
#pragma unroll
    for (int e = 0; e < V; ++e) {
      hb[e] = float_to_bf16_bits(v[e]);
      lb[e] = float_to_bf16_bits(v[e] - bf16_bits_to_float(hb[e]));
    }
    if constexpr (V == 1) {
      uhi[lane] = hb[0];
      ulo[lane] = lb[0];
    } else {
      uint32_t hw[V / 2], lw[V / 2];
#pragma unroll
      for (int i = 0; i < V / 2; ++i) {
        hw[i] = (uint32_t)hb[2 * i] | ((uint32_t)hb[2 * i + 1] << 16);
        lw[i] = (uint32_t)lb[2 * i] | ((uint32_t)lb[2 * i + 1] << 16);
      }
      if constexpr (V == 8) {
        reinterpret_cast<uint4*>(uhi)[lane] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        reinterpret_cast<uint4*>(ulo)[lane] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
      } else if constexpr (V == 4) {
        reinterpret_cast<uint2*>(uhi)[lane] = make_uint2(hw[0], hw[1]);
        reinterpret_cast<uint2*>(ulo)[lane] = make_uint2(lw[0], lw[1]);
      } else {
        reinterpret_cast<uint32_t*>(uhi)[lane] = hw[0];
        reinterpret_cast<uint32_t*>(ulo)[lane] = lw[0];
      }
    }
  }
  return mx;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}

// x_tilde = D^T u of the polyphase build, for B a compile-time constant:
// warp items (16-row tile rt of (m, b) rows, code tiles jt, jt + 1), 16-deep
// steps s over the inputs in natural order.  A = u hi and lo rows by
// ldmatrix; code row j = r + p m takes taps D^T[r][(i - q m) mod B] for
// i = 16 s + 2t (+1, +8, +9) at table entry jbase[j] + 2t + 16 s (+8): one
// base per lane and tile, constant offsets per step.  u hi D hi, u lo D hi
// and u hi D lo go to three accumulators (short dependency chains); the
// lo x lo term is below fp32 rounding of the sum.  rowoff / rowxm give each
// (m, b) row's chunk-local first code and scratch offset (rowoff is far
// negative for rows past the chunk's).
template <int B>
__device__ __forceinline__ void poly_items(const DecodeParams& p, const BuildGeo& q, float* xs,
                                           const uint16_t* uhi, const uint16_t* ulo, const uint2* ptab,
                                           const int* jbase, const int* rowoff, const int* rowxm, int ew, int lane) {
  constexpr int S = B / 16, US = B + 8, NW = kBuildThreads / 32;
  const int g = lane >> 2, t = lane & 3;
  const int JT = p.n_b / 8, JP = (JT + 1) / 2, RT = (q.rows + 15) / 16;
  const bool ter = p.ternary != 0;
  const int lim = (int)(q.k1 - q.k0);
  const int lrow = (lane & 7) + 8 * ((lane >> 3) & 1), lcol = 8 * (lane >> 4);   // ldmatrix row of this lane
  for (int it = ew; it < RT * JP; it += NW) {
    const int rt = it < JP ? 0 : it / JP, jt = 2 * (it - rt * JP);
    const bool two = jt + 1 < JT;
    const uint32_t ah_at = smem_u32(uhi + (rt * 16 + lrow) * US + lcol);
    const uint32_t al_at = smem_u32(ulo + (rt * 16 + lrow) * US + lcol);
    const uint2* pb0 = ptab + jbase[8 * jt + g] + 2 * t;
    const uint2* pb1 = ptab + (two ? jbase[8 * jt + 8 + g] : 0) + 2 * t;
    float h0[4] = {0.f, 0.f, 0.f, 0.f}, a0[4] = {0.f, 0.f, 0.f, 0.f}, b0[4] = {0.f, 0.f, 0.f, 0.f};
    float h1[4] = {0.f, 0.f, 0.f, 0.f}, a1[4] = {0.f, 0.f, 0.f, 0.f}, b1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int s = 0; s < S; ++s) {
      uint32_t ah[4], al[4];
      ldsm_x4(ah_at + 32 * s, ah);
      ldsm_x4(al_at + 32 * s, al);
      const uint2 e0 = pb0[16 * s], f0 = pb0[16 * s + 8];
      mma_bf16_16816(h0, ah, e0.x, f0.x);
      mma_bf16_16816(a0, al, e0.x, f0.x);
      mma_bf16_16816(b0, ah, e0.y, f0.y);
      if (two) {
        const uint2 e1 = pb1[16 * s], f1 = pb1[16 * s + 8];
        mma_bf16_16816(h1, ah, e1.x, f1.x);
        mma_bf16_16816(a1, al, e1.x, f1.x);
        mma_bf16_16816(b1, ah, e1.y, f1.y);
      }
    }
    // accumulator element e: (m, b) row rt 16 + g + 8 (e >> 1), code 8 jt + 2t + (e & 1)
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int rho = rt * 16 + g + 8 * hh;
      const int off = rowoff[rho] + 8 * jt + 2 * t;   // chunk-local code
      float* xm = xs + rowxm[rho];
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int tile = 0; tile < 2; ++tile) {
          if (tile == 1 && !two) continue;
          const int kl = off + 8 * tile + c, e = 2 * hh + c;
          if ((unsigned)kl >= (unsigned)lim) continue;
          const float v = tile ? h1[e] + (a1[e] + b1[e]) : h0[e] + (a0[e] + b0[e]);
          xm[(kl >> 7) * kXtStride + decode_pos(kl & 127, ter)] = v;
        }
    }
  }
}

__device__ __forceinline__ int term_exponent(float mx, float gnorm) {
  int e = 0;
  if (mx > 0.f) {   // bound = mx gnorm < 2^(e1 + e2) without forming it (no overflow)
    int e1 = 0, e2 = 0;
    frexpf(mx, &e1);
    frexpf(gnorm, &e2);
    e = e1 + e2 - 8;   // bound * 2^-e < 256 < 448
  }
  return max(e, -120);
}

// Called by the kBuildThreads expander threads before their first stage; it
// waits for the preceding grid itself (x may come from it; G does not).
__device__ void build_b_operand(const DecodeParams& p, uint8_t* bop, float* xs, int kb0, int ncb, int et,
                                uint32_t* xmax_u, float* inv_s, float* scale_s) {
  BuildGeo q;
  q.k0 = (int64_t)kb0 * kBlk;
  q.kend = q.k0 + (int64_t)ncb * kBlk;
  q.k1 = min(q.kend, p.k_eff);
  q.blo = (int)(q.k0 / p.n_b);
  q.nbi = (int)((q.k1 - 1) / p.n_b) - q.blo + 1;   // k1 > k0: a block always holds a code
  q.rows = p.M * q.nbi;
  q.kbw = g_frag_batch(p.B);
  q.R = q.kbw / 4;
  q.nkb = p.B / q.kbw;
  q.S4 = q.kbw / 16;
  const int ew = et >> 5, lane = et & 31, g = lane >> 2, t = lane & 3;
  constexpr int NW = kBuildThreads / 32;
  const int JT = p.n_b / 8;

  if (p.use_poly) {
    // Polyphase build.  The table goes to shared memory before the wait (a
    // plan constant); then each warp transforms (m, b) rows u = Had^T x_b
    // (bf16 hi + lo rows behind the fp32 scratch) and adds max |x| into
    // xmax_u; after one barrier the warps take (row tile, code tile pair)
    // items of x_tilde = D^T u on warp MMAs.
    const int B = p.B, us = B + 8, RT = (q.rows + 15) / 16;
    uint16_t* uhi = reinterpret_cast<uint16_t*>(xs + (size_t)p.M * p.CB * kXtStride);
    uint16_t* ulo = uhi + (size_t)16 * RT * us;
    uint2* ptab = reinterpret_cast<uint2*>(ulo + (size_t)16 * RT * us);
    int* jbase = reinterpret_cast<int*>(ptab + p.poly_bytes / 8);   // n_b entries
    int* rowoff = jbase + p.n_b;                                      // 16 RT (m, b) rows
    int* rowxm = rowoff + 16 * RT;
    for (int i = et; i < p.poly_bytes / 16; i += kBuildThreads)
      reinterpret_cast<uint4*>(ptab)[i] = __ldg(reinterpret_cast<const uint4*>(p.poly) + i);
    for (int j = et; j < p.n_b; j += kBuildThreads)   // code row j = r + p m: phase row r, taps from -q m
      jbase[j] = (j % p.poly_p) * poly_stride(B) + ((-p.poly_q * (j / p.poly_p)) & (B - 1));
    pdl_wait();
    const int V = B >= 32 ? B / 32 : 1;
    for (int rho = ew; rho < 16 * RT; rho += NW) {
      const bool in = rho < q.rows;
      const int m = in ? rho / q.nbi : 0;
      const bool act = in && lane * V < B;
      const uint16_t* xr = p.x + (size_t)m * p.K + (size_t)(q.blo + rho - m * q.nbi) * B + lane * V;
      uint16_t* rh = uhi + (size_t)rho * us;
      uint16_t* rl = ulo + (size_t)rho * us;
      float mx;
      switch (V) {
        case 8: mx = row_transform<8>(p, xr, act, lane, rh, rl); break;
        case 4: mx = row_transform<4>(p, xr, act, lane, rh, rl); break;
        case 2: mx = row_transform<2>(p, xr, act, lane, rh, rl); break;
        default: mx = row_transform<1>(p, xr, act, lane, rh, rl); break;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) {
        if (in) atomicMax(xmax_u + m, __float_as_uint(mx));   // non-negative: integer order
        rowoff[rho] = in ? (q.blo + rho - m * q.nbi) * p.n_b - (int)q.k0 : -(1 << 30);
        rowxm[rho] = m * ncb * kXtStride;
      }
    }
    named_bar_sync(3, kBuildThreads);
    if (et < p.M) {
      const int e = term_exponent(__uint_as_float(xmax_u[et]), p.gnorm);
      scale_s[et] = ldexpf(1.f, e);
      inv_s[et] = ldexpf(1.f, -e);
    }
    switch (B) {
      case 16: poly_items<16>(p, q, xs, uhi, ulo, ptab, jbase, rowoff, rowxm, ew, lane); break;
      case 32: poly_items<32>(p, q, xs, uhi, ulo, ptab, jbase, rowoff, rowxm, ew, lane); break;
      case 64: poly_items<64>(p, q, xs, uhi, ulo, ptab, jbase, rowoff, rowxm, ew, lane); break;
      case 128: poly_items<128>(p, q, xs, uhi, ulo, ptab, jbase, rowoff, rowxm, ew, lane); break;
      default: poly_items<256>(p, q, xs, uhi, ulo, ptab, jbase, rowoff, rowxm, ew, lane); break;
    }
  } else {
    pdl_wait();
    // max |x[m, .]| over the chunk's input blocks: 16-byte loads, 4 in flight
    const int bq = p.B / 8;
    const int nq = q.rows * bq;
    for (int i0 = et; i0 < nq; i0 += 4 * kBuildThreads) {
      uint4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * kBuildThreads;
        v[u] = make_uint4(0, 0, 0, 0);
        if (i < nq) {
          const int rho = i / bq, c = i - rho * bq, m = rho / q.nbi, b = q.blo + rho - m * q.nbi;
          v[u] = __ldg(reinterpret_cast<const uint4*>(p.x + (size_t)m * p.K + (size_t)b * p.B) + c);
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * kBuildThreads;
        if (i < nq) {
          const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
          float mx = 0.f;
#pragma unroll
          for (int c = 0; c < 4; ++c) mx = fmaxf(mx, fmaxf(bf16_mag(w[c]), bf16_mag(w[c] >> 16)));
          atomicMax(xmax_u + (i / bq) / q.nbi, __float_as_uint(mx));   // non-negative floats order as integers
        }
      }
    }
    named_bar_sync(3, kBuildThreads);
    if (et < p.M) {
      const int e = term_exponent(__uint_as_float(xmax_u[et]), p.gnorm);
      scale_s[et] = ldexpf(1.f, e);
      inv_s[et] = ldexpf(1.f, -e);
    }
    named_bar_sync(3, kBuildThreads);
    const int RT = (q.rows + 15) / 16;
    for (int it = ew; it < RT * JT; it += NW) {
      const int rt = it / JT, jt = it - rt * JT;
      const int r0 = rt * 16 + g, r1 = r0 + 8;
      const int m0 = r0 < q.rows ? r0 / q.nbi : 0, m1 = r1 < q.rows ? r1 / q.nbi : 0;
      const uint16_t* xa0 = p.x + t * q.R + (r0 < q.rows ? (size_t)m0 * p.K + (size_t)(q.blo + r0 - m0 * q.nbi) * p.B : 0);
      const uint16_t* xa1 = p.x + t * q.R + (r1 < q.rows ? (size_t)m1 * p.K + (size_t)(q.blo + r1 - m1 * q.nbi) * p.B : 0);
      float acc4[2][4] = {};
      for (int kb = 0; kb < q.nkb; ++kb) {
        uint32_t xw[2][8], gw[16];
        load_x_frags(q, xa0, xa1, kb, xw);
        load_g_frags(p, q, jt, kb, lane, gw);
        mma_batch(q, xw, gw, acc4);
      }
      float acc[4];
      acc_sum(acc4, acc);
      store_xt(p, q, xs, ncb, jt, t, r0, r1, m0, m1, acc);
    }
  }
  // x_tilde (all of the chunk, in the scratch) -> e4m3 terms: one thread per
  // (m, block, 16-position chunk), 16-byte stores, consecutive threads on
  // consecutive chunks of a term row (no bank conflicts); per half chunk, 8-byte
  // stores, when whole chunks would leave half the builders idle.
  named_bar_sync(3, kBuildThreads);
  const int lim = (int)(q.k1 - q.k0);
  if (p.M * ncb * 8 <= kBuildThreads / 2)   // too few 16-position tasks for the builders: halve them
    all_terms<8>(p, bop, xs, ncb, et, inv_s, lim);
  else
    all_terms<16>(p, bop, xs, ncb, et, inv_s, lim);
  fence_proxy_async_smem();   // generic-proxy stores -> the MMAs' async-proxy reads
  named_bar_sync(3, kBuildThreads);
}

// kStream: the B operand comes with each stage (p.stream); one instantiation
// per mode keeps the resident mode's code free of the streamed bookkeeping.
template <bool kStream>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(DecodeParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t c_full[kMaxRing], c_empty[kMaxRing];
  __shared__ __align__(8) uint64_t a_full[2 * kSlots], a_empty[2 * kSlots];
  __shared__ __align__(8) uint64_t acc_full[2][2], acc_empty[2][2], b_full, mma_done[2];
  __shared__ uint32_t tmem_base;
  __shared__ int last[1];
  __shared__ uint32_t red_bits[kRedWords];  // tiles whose split-K sum this CTA owes (all threads sum)
  __shared__ float scale_s[kMaxDecodeM];   // 2^e_m
  __shared__ float inv_s[kMaxFuseM];       // 2^-e_m (fused B operand)
  __shared__ uint32_t xmax_u[kMaxFuseM];   // max |x[m]| bits (fused B operand)
  __shared__ int sblk[kMaxSpu + 1];         // first block of stage j of a tile

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int sidx = blockIdx.x % p.S, prow = blockIdx.x / p.S;
  const int kb0 = sidx * p.CB;
  const int ncb = min(p.CB, p.KB - kb0);                        // blocks of this chunk
  const int spu = max((ncb + p.sb - 1) / p.sb, min(2, ncb));   // stages per tile
  const int nunits = (p.ntiles - prow + p.P - 1) / p.P;         // row tiles of this CTA
  // The CTAs of a row set (one per k chunk) walk its tiles in rotated orders,
  // so that a different CTA finishes (and sums the split-K partials of) each
  // tile: unit u is tile prow + ((u + rot) mod nunits) P.  (In one common
  // order, a CTA that runs slightly behind the others arrives last on every
  // tile and sums them all: at M = 1 that added ~20 us to 8192 x 28672.)
  const bool red_now = p.M == 1;
  const int rot = (int)(((int64_t)sidx * ((nunits + p.S - 1) / p.S)) % max(nunits, 1));
  const int nstages = nunits * spu;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* bop = base;                                          // ncb x NP x 128 bytes
  uint8_t* ring = base + p.b_bytes;                             // ring x slot_bytes

  // Set-up spread over warps 1.. (warp 0 allocates TMEM meanwhile).
  if (warp == 1 && lane < p.ring) {
    mbar_init(&c_full[lane], 1);
    mbar_init(&c_empty[lane], kStream ? 5 : 4);   // one arrival per expander warp (+ the MMAs' commit)
  } else if (warp == 2) {
    if (lane < 2 * kSlots) {
      mbar_init(&a_full[lane], 4);
      mbar_init(&a_empty[lane], 1);
    } else if (lane < 2 * kSlots + 4) {
      const int e = (lane - 2 * kSlots) >> 1, b = lane & 1;
      mbar_init(&acc_full[e][b], 1);
      mbar_init(&acc_empty[e][b], 128);
    } else if (lane == 2 * kSlots + 4) {
      mbar_init(&b_full, 1);
    } else if (lane == 2 * kSlots + 5 || lane == 2 * kSlots + 6) {
      mbar_init(&mma_done[lane - 2 * kSlots - 5], 1);
    } else if (lane >= 16 && lane < 16 + kMaxFuseM) {
      xmax_u[lane - 16] = 0u;
    }
  } else if (warp >= 3 && warp < 3 + (kMaxSpu + 32) / 32) {
    const int j = tid - 96;
    if (j <= spu) sblk[j] = stage_block(j, ncb, spu);
  } else if (warp >= 8 && warp < 10) {
    red_bits[tid - 256] = 0u;
  }
  if (warp == 1 || warp == 2) fence_mbar_init();
  if (warp == 0) {
    __syncwarp();
    tmem_alloc(&tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_launch_dependents();
  // (the B operand builders of the fused path wait inside build_b_operand)
  const bool builder = p.fused && warp >= kExpWarp0 && warp < kEpiWarp0;
  if (!builder && (warp >= kProducers || !p.early)) pdl_wait();
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp < kProducers) {
    if (lane == 0) {
      // Producer of pipeline `warp`: stages i = warp (mod 2), ring slots
      // i mod ring (ring is even).  Stage (unit u, j) is the
      // slabs (tile, 2 b) .. (tile, 2 b' - 1) of its blocks [b, b'),
      // adjacent in the tiled layout.  Producer 0 also copies the chunk's B
      // operand: after its first two stages when the codes may be read before
      // the preceding grid is done, before everything otherwise.
      int last_i = -1;
      bool b_loaded = warp != 0 || p.fused || kStream;   // fused: the expanders build it
      if (kStream && warp == 0) mbar_arrive(&b_full);   // streamed: nothing resident to wait for
      // Fused: the first kFusePre stages go out at once, the rest once the B
      // operand is built, so that the builders' loads do not queue behind a
      // full ring of code copies.
      bool b_ready = !p.fused;
      const int pre = p.early ? min(2 * kProducers, nstages) : 0;
      int u = 0, j = warp;
      while (j >= spu) { j -= spu; ++u; }
      const uint64_t pol = l2_policy_evict_first();   // codes are read once per call
      for (int i = warp; i < nstages && ok; i += kProducers) {
        if (!b_loaded && i >= pre) {
          if (p.early) pdl_wait();
          mbar_expect_tx(&b_full, p.b_bytes);
          bulk_g2s(bop, p.bimg + (size_t)kb0 * p.NP * 128, p.b_bytes, &b_full);
          b_loaded = true;
        }
        if (!b_ready && i >= kFusePre) {
          ok = mbar_wait(&b_full, 0);
          if (!ok) break;
          b_ready = true;
        }
        const int slot = i % p.ring, r = i / p.ring;
        if (r > 0) ok = mbar_wait(&c_empty[slot], (r - 1) & 1);
        if (!ok) break;
        const int b0 = sblk[j], b1 = sblk[j + 1];
        const int tile = prow + (u + rot < nunits ? u + rot : u + rot - nunits) * p.P;
        const uint8_t* src = reinterpret_cast<const uint8_t*>(p.codes) +
                             ((size_t)tile * p.KB + kb0 + b0) * p.blk_bytes;
        const uint32_t bytes = (uint32_t)(b1 - b0) * p.blk_bytes;
        uint8_t* dst = ring + (size_t)slot * p.slot_bytes;
        if constexpr (kStream) {   // the stage's B rows behind the slot's code area
          const uint32_t bb = (uint32_t)(b1 - b0) * p.NP * 128;
          mbar_expect_tx(&c_full[slot], bytes + bb);
          bulk_g2s_hint(dst, src, bytes, &c_full[slot], pol);
          bulk_g2s(dst + (size_t)p.sb * p.blk_bytes, p.bimg + (size_t)(kb0 + b0) * p.NP * 128, bb, &c_full[slot]);
        } else {
          mbar_expect_tx(&c_full[slot], bytes);
          bulk_g2s_hint(dst, src, bytes, &c_full[slot], pol);
        }
        last_i = i;
        j += kProducers;
        while (j >= spu) { j -= spu; ++u; }
      }
      if (!b_loaded) {   // producer 0 had no stage at or past `pre`, or failed
        if (p.early) pdl_wait();
        if (ok) {
          mbar_expect_tx(&b_full, p.b_bytes);
          bulk_g2s(bop, p.bimg + (size_t)kb0 * p.NP * 128, p.b_bytes, &b_full);
        }
        b_loaded = ok;
      }
      // Every copy this thread issued has landed before the CTA may exit.
      if (warp == 0 && !p.fused && b_loaded && !mbar_wait(&b_full, 0)) ok = false;
      for (int i = last_i; i >= 0 && i > last_i - p.ring; i -= kProducers)
        if (!mbar_wait(&c_full[i % p.ring], (i / p.ring) & 1)) ok = false;
    }
  } else if (warp < kExpWarp0) {
    if (lane == 0) {
      // MMA issuer of pipeline e: stages i = e (mod 2), the pipeline's jj-th
      // stage (jj = i / 2) in TMEM slot 2e + (jj mod 2), into its own
      // accumulator.
      const int e = warp - kIssuerWarp0;
      ok = mbar_wait(&b_full, 0);
      tc_fence_after();
      // kind::f8f6f4: D fp32, A and B e4m3, both K-major, N = NP, M = 128.
      const uint32_t idesc = (1u << 4) | ((uint32_t)(p.NP >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
      // Per stage: one wait, 4 nb MMAs, one commit; stage bookkeeping is
      // kept incremental (a single thread's scalar latency is on the path).
      const uint64_t bd0 = sw128_desc(sbase);
      const uint64_t bstep = (uint64_t)((p.NP * 128) >> 4);   // descriptor units per block
      const uint32_t abase = tmem + (uint32_t)(kSlots * e * 32 * p.sb);
      const uint32_t aslot = (uint32_t)(32 * p.sb);
      int k = 0, buf = 0, u = 0, j = e;
      while (j >= spu) { j -= spu; ++u; }
      bool first = true;
      uint32_t dt = 0;
      int last_c = -1;   // last stage whose slot this thread released by commit
      // streamed: B rows of stage i in ring slot i mod ring, behind its codes
      const uint64_t sd0 = sw128_desc(sbase + p.b_bytes + (uint32_t)p.sb * p.blk_bytes);
      const uint64_t sstep = (uint64_t)(p.slot_bytes >> 4);
      int slot = e;
      for (int i = e, jj = 0; i < nstages && ok; i += 2, ++jj) {
        if (first) {
          buf = p.nbuf == 2 ? (k & 1) : 0;
          if (k >= p.nbuf) {
            ok = mbar_wait(&acc_empty[e][buf], ((k / p.nbuf) - 1) & 1);
            if (!ok) break;
          }
          dt = tmem + (uint32_t)(p.dbase + (e * p.nbuf + buf) * p.NP);
        }
        const int a = kSlots * e + (jj & 1);
        ok = mbar_wait(&a_full[a], (jj >> 1) & 1);
        if (!ok) break;
        tc_fence_after();
        const int b0 = sblk[j], nb = sblk[j + 1] - b0;
        uint64_t bd;
        if constexpr (kStream) bd = sd0 + (uint64_t)slot * sstep;
        else bd = bd0 + (uint64_t)b0 * bstep;
        uint32_t at = abase + (uint32_t)(jj & 1) * aslot;
        for (int bb = 0; bb < nb; ++bb, at += 32, bd += bstep) {
          umma_f8_ts(dt, at, bd, idesc, (first && bb == 0) ? 0u : 1u);
          umma_f8_ts(dt, at + 8, bd + 2, idesc, 1u);
          umma_f8_ts(dt, at + 16, bd + 4, idesc, 1u);
          umma_f8_ts(dt, at + 24, bd + 6, idesc, 1u);
        }
        umma_commit(&a_empty[a]);
        if constexpr (kStream) {   // the slot's B rows are free once these MMAs are done
          umma_commit(&c_empty[slot]);
          last_c = i;
          slot += 2;
          if (slot >= p.ring) slot -= p.ring;
        }
        const int u0 = u;
        j += 2;
        while (j >= spu) { j -= spu; ++u; }
        first = u != u0;
        if (first) {   // this pipeline's last stage of the tile
          umma_commit(&acc_full[e][buf]);
          ++k;
        }
      }
      umma_commit(&mma_done[e]);   // every MMA issued has finished before TMEM is freed
      if (!mbar_wait(&mma_done[e], 0)) ok = false;
      // ... and the last commit to each of this pipeline's TMEM slots has
      // arrived (those phases have no other waiter).
      const int njs = (nstages - e + 1) / 2;   // stages of this pipeline
      for (int jj = max(0, njs - kSlots); jj < njs; ++jj)
        if (!mbar_wait(&a_empty[kSlots * e + jj % kSlots], (jj / kSlots) & 1)) ok = false;
      // Streamed B: the slot commits of the last stages, which no producer
      // waits for (the expanders arrived before these stages' MMAs).
      for (int i = last_c; i >= 0 && i + p.ring >= nstages; i -= 2)
        if (!mbar_wait(&c_empty[i % p.ring], (i / p.ring) & 1)) ok = false;
    }
  } else if (warp < kEpiWarp0) {
    // ------------------------------------------------------------ expanders
    // Set x = 2e + t expands stages i = e + 2t (mod 4) in order: TMEM slot
    // x, ring slots i mod ring (ring is a multiple of 4).
    if (p.fused) {
      // scratch: the ring slots the first kFusePre stages do not use
      float* xs = reinterpret_cast<float*>(ring + (size_t)kFusePre * p.slot_bytes);
      build_b_operand(p, bop, xs, kb0, ncb, tid - 32 * kExpWarp0, xmax_u, inv_s, scale_s);
      if (tid == 32 * kExpWarp0) mbar_arrive(&b_full);
    }
    const int x = (warp - kExpWarp0) >> 2, q = warp & 3, r = 32 * q + lane;
    const int ex = x / kSlots, tx = x - ex * kSlots;
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * q) << 16);
    const uint32_t slab = p.blk_bytes / 2;
    int u = 0, j = ex + 2 * tx;
    while (j >= spu) { j -= spu; ++u; }
    for (int i = ex + 2 * tx; i < nstages && ok; i += 2 * kSlots) {
      const int slot = i % p.ring, jj = i >> 1, a = x;
      ok = warp_wait(&c_full[slot], (i / p.ring) & 1);
      if (!ok) break;
      // Codes into registers first, so that the ring slot goes back to the
      // producer before this set waits for its TMEM slot.
      const int nb = sblk[j + 1] - sblk[j];
      j += 2 * kSlots;
      while (j >= spu) { j -= spu; ++u; }
      const uint8_t* cs = ring + (size_t)slot * p.slot_bytes;
      uint32_t w[kMaxSb][8];
#pragma unroll
      for (int bb = 0; bb < kMaxSb; ++bb) {
        if (bb < nb) {
          const uint8_t* cb = cs + bb * p.blk_bytes;
          if (p.ternary) {
            const uint4 g0 = *reinterpret_cast<const uint4*>(cb + r * 16);
            const uint4 g1 = *reinterpret_cast<const uint4*>(cb + slab + r * 16);
            w[bb][0] = g0.x; w[bb][1] = g0.y; w[bb][2] = g0.z; w[bb][3] = g0.w;
            w[bb][4] = g1.x; w[bb][5] = g1.y; w[bb][6] = g1.z; w[bb][7] = g1.w;
          } else {
            const uint2 g0 = *reinterpret_cast<const uint2*>(cb + r * 8);
            const uint2 g1 = *reinterpret_cast<const uint2*>(cb + slab + r * 8);
            w[bb][0] = ~g0.x; w[bb][1] = ~g0.y; w[bb][2] = ~g1.x; w[bb][3] = ~g1.y;
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&c_empty[slot]);
      if (jj >= kSlots) {
        ok = warp_wait(&a_empty[a], ((jj / kSlots) - 1) & 1);
        if (!ok) break;
        tc_fence_after();
      }
#pragma unroll
      for (int bb = 0; bb < kMaxSb; ++bb) {
        if (bb < nb) {
          uint32_t v[32];
          if (p.ternary) {
#pragma unroll
            for (int wi = 0; wi < 8; ++wi)
#pragma unroll
              for (int jb = 0; jb < 4; ++jb) v[4 * wi + jb] = (w[bb][wi] << (2 * jb)) & 0xC0C0C0C0u;
          } else {
#pragma unroll
            for (int wi = 0; wi < 4; ++wi)
#pragma unroll
              for (int jb = 0; jb < 8; ++jb) v[8 * wi + jb] = ((w[bb][wi] << jb) & 0x80808080u) | 0x40404040u;
          }
          tmem_st32(lane_addr + (uint32_t)(a * 32 * p.sb + 32 * bb), v);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[a]);
    }
  } else {
    // ------------------------------------------------------------- epilogue
    const int q = warp & 3, r = 32 * q + lane, et = tid - 32 * kEpiWarp0;
    const int NR = p.ntiles * kTileRows;
    const int MT = p.M * p.T;
    // a split-K sum costs M x ceil(S / 16) rounds of 16 loads per thread
    auto reduce_tile = [&](int ut) {
      const int row = (prow + ut * p.P) * kTileRows + r;
      if (row >= p.n_out) return;
      const float sa = 0.5f * __ldg(p.alpha + row);
      const size_t sstride = (size_t)p.M * NR;
      for (int mm = 0; mm < p.M; ++mm) {
        const float* pr = p.part + (size_t)mm * NR + row;
        float s0 = 0.f;
        for (int k0 = 0; k0 < p.S; k0 += 16) {   // 16 loads in flight, summed in chunk order
          float a[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) a[i] = k0 + i < p.S ? __ldcg(pr + (size_t)(k0 + i) * sstride) : 0.f;
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (k0 + i < p.S) s0 += a[i];
        }
        p.y[(size_t)mm * p.n_out + row] = sa * s0;
      }
    };
    call_record_start(p.rec, p.call, blockIdx.x == 0 && et == 0);
    if (p.fused) {   // scale_s was written by the B operand builders
      ok = group_and(2, 128, mbar_wait(&b_full, 0));
    } else {
      if (et < p.M) scale_s[et] = ldexpf(1.f, p.sexp[et]);
      named_bar_sync(2, 128);
    }
    int kc[2] = {0, 0};
    for (int u = 0; u < nunits && ok; ++u) {
      // issuers with stages in this tile: both, unless the tile is one stage
      const bool in0 = spu >= 2 || ((u * spu) & 1) == 0;
      const bool in1 = spu >= 2 || ((u * spu) & 1) == 1;
      const int bf0 = kc[0] % p.nbuf, bf1 = kc[1] % p.nbuf;
      bool w = true;
      if (in0) w = mbar_wait(&acc_full[0][bf0], (kc[0] / p.nbuf) & 1);
      if (in1 && w) w = mbar_wait(&acc_full[1][bf1], (kc[1] / p.nbuf) & 1);
      ok = group_and(2, 128, w);
      if (!ok) break;
      tc_fence_after();
      const int ut = u + rot < nunits ? u + rot : u + rot - nunits;   // unit of this tile
      const int row = (prow + ut * p.P) * kTileRows + r;
      const bool live = row < p.n_out;
      const float sa = live ? 0.5f * __ldg(p.alpha + row) : 0.f;
      const uint32_t lq = tmem + ((uint32_t)(32 * q) << 16);
      const uint32_t d0 = lq + (uint32_t)(p.dbase + bf0 * p.NP);
      const uint32_t d1 = lq + (uint32_t)(p.dbase + (p.nbuf + bf1) * p.NP);
      int m = 0, t = 0;
      float acc = 0.f, wt = 1.f;
      for (int c0 = 0; c0 < MT; c0 += 16) {
        uint32_t r0[16], r1[16];
        if (in0) tmem_ld16(d0 + (uint32_t)c0, r0);
        if (in1) tmem_ld16(d1 + (uint32_t)c0, r1);
        tmem_ld_wait();
        if (c0 + 16 >= MT) {
          tc_fence_before();
          if (in0) mbar_arrive(&acc_empty[0][bf0]);
          if (in1) mbar_arrive(&acc_empty[1][bf1]);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          if (c0 + i < MT) {
            const float dv = (in0 ? __uint_as_float(r0[i]) : 0.f) + (in1 ? __uint_as_float(r1[i]) : 0.f);
            acc += wt * dv;
            wt *= 0.0625f;
            if (++t == p.T) {
              const float ym = acc * scale_s[m];
              if (p.S == 1) {
                if (live) p.y[(size_t)m * p.n_out + row] = sa * ym;
              } else {
                p.part[((size_t)sidx * p.M + m) * NR + row] = ym;
              }
              acc = 0.f; wt = 1.f; t = 0; ++m;
            }
          }
        }
      }
      kc[0] += in0;
      kc[1] += in1;
      if (p.S > 1) {
        // Split-K, per tile while the next tile's MMAs run: one thread takes
        // the tile's ticket (after the barrier that orders the other threads'
        // partial stores before the ticket's release fence); the CTA with the
        // last ticket fences again and sums the S partials in k-chunk order
        // (deterministic): at once for M = 1, else after the main loop on all
        // of the CTA's threads (the tiles a CTA finishes last come at the end
        // of its rotated order).
        named_bar_sync(2, 128);
        if (et == 0) {
          const uint32_t n = ticket_take(p.cnt + prow + ut * p.P, p.call);
          if (n == 0) call_record_fail(p.rec, p.call);
          const bool won = n == (uint32_t)p.S;
          if (won) fence_acq_rel_gpu();
          const bool defer = won && !red_now && ut < 32 * kRedWords;
          if (defer) red_bits[ut >> 5] |= 1u << (ut & 31);
          last[0] = won && !defer;
        }
        named_bar_sync(2, 128);
        if (last[0]) reduce_tile(ut);
      }
    }
  }
  if (!ok) call_record_fail(p.rec, p.call);
  tc_fence_before();
  __syncthreads();
  // Split-K sums won in the end-of-kernel ticket burst, by every thread of the
  // CTA: (m, row) pairs, consecutive threads on consecutive rows; each pair
  // adds its S partials in k-chunk order (deterministic) with 16 loads in
  // flight.
  if (p.S > 1 && ok && !red_now) {
    const int NR = p.ntiles * kTileRows;
    const size_t sstride = (size_t)p.M * NR;
    for (int w = 0; w < kRedWords; ++w) {
      uint32_t bits = red_bits[w];
      while (bits) {
        const int u = 32 * w + __ffs(bits) - 1;
        bits &= bits - 1;
        const int row0 = (prow + u * p.P) * kTileRows;
        for (int i = tid; i < kTileRows * p.M; i += kThreads) {
          const int mm = i / kTileRows, row = row0 + (i - mm * kTileRows);
          if (row >= p.n_out) continue;
          const float* pr = p.part + (size_t)mm * NR + row;
          float s0 = 0.f;
          for (int k0 = 0; k0 < p.S; k0 += 16) {
            float a[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) a[j] = k0 + j < p.S ? __ldcg(pr + (size_t)(k0 + j) * sstride) : 0.f;
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (k0 + j < p.S) s0 += a[j];
          }
          p.y[(size_t)mm * p.n_out + row] = 0.5f * __ldg(p.alpha + row) * s0;
        }
      }
    }
  }
  if (warp == 0) {
    __syncwarp();   // warp-collective: lane 0 ran the producer loop alone
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// TMEM split for N = NP: accumulators (2 pipelines x nbuf buffers x NP
// columns) at the top, four A slots of sb blocks (32 sb columns) below.
void tmem_split(int NP, int* sb, int* nbuf, int* dbase) {
  *nbuf = NP <= 32 ? 2 : 1;
  const int dcols = 2 * *nbuf * NP;
  *sb = std::max(1, std::min(kMaxSb, (512 - dcols) / (2 * kSlots * 32)));
  *dbase = 512 - dcols;
}

}  // namespace

// Launch shape for batch M: the (S, P) grid of at most one CTA per SM that
// minimises a simple time model: the larger of the MMA time of the busiest
// CTA and the HBM time of codes plus split-K partials (the bytes in flight
// capped by the CTAs' code rings), plus the split-K tail (one fence, one
// ticket, the final sums).
DecodeConfig decode_config_search(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  DecodeConfig best{};
  best.M = M;
  best.T = decode_terms(M);
  best.NP = (M * best.T + 15) / 16 * 16;
  const int KB = (int)(g.k_eff_pad / kBlk);
  const int sms = std::max(1, pl->sm_count);
  const int blk_bytes = kTileRows * kBlk * g.bits / 8;
  int sb = 0, nbuf = 0, dbase = 0;
  tmem_split(best.NP, &sb, &nbuf, &dbase);
  const int slot_bytes = sb * blk_bytes;
  // M = 1 constants fitted to measured launches: each split-K tile costs
  // its epilogue (partial stores, a release fence and a ticket round trip
  // while the code stream loads HBM) beyond its MMAs, and the ring's copies
  // see a longer loaded latency.  Fewer, longer tiles per CTA measured
  // faster both alone and inside the 7-linear layer step (8192 x 8192:
  // S = 4 instead of 9, 31.0 -> 27.5 us per launch); for 8192 x 28672 the
  // configurations that were faster alone were slower inside the step, and
  // these constants keep S = 19 there.  Larger batches keep the earlier
  // constants.
  const double clk = 1.9e9, bw = 6.5e12;
  const double latency = M == 1 ? 3.0e-6 : 2.2e-6;             // loaded HBM latency
  const double t_tile = M == 1 ? 0.5e-6 : 0.0;                 // per split-K tile
  const double t_mma = std::max(38.0, best.NP * 0.55) / clk;    // per MMA, two issuers
  const double code_bytes = (double)g.ntiles * kTileRows * g.k_eff_pad * g.bits / 8;
  double best_t = 1e30;
  // Streamed B (batches past the one-kernel route): each stage's slot holds
  // its blocks' B rows too, so chunks are not bounded by a resident image
  // and the split-K partials (S M N floats) can stay small.
  const int nmode = M > kMaxFuseM ? 2 : 1;
  for (int stream = 0; stream < nmode; ++stream)
  for (int S = 1; S <= std::min(KB, sms); ++S) {
    const int CB = (KB + S - 1) / S;
    if ((S - 1) * CB >= KB) continue;                      // no empty chunk
    const int b_bytes = stream ? 0 : CB * best.NP * 128;
    const int sbytes = stream ? sb * (blk_bytes + best.NP * 128) : slot_bytes;
    int ring = std::min(kMaxRing, (kSmemMax - 2048 - b_bytes) / sbytes);
    ring -= ring % kExpSets;          // each ring slot belongs to one expander set
    if (ring < kExpSets) continue;
    const int spu = std::max((CB + sb - 1) / sb, std::min(2, CB));
    if (spu > kMaxSpu) continue;
    for (int P = 1; P <= std::min(g.ntiles, sms / S); ++P) {
      const int grid = S * P;
      const int units = (g.ntiles + P - 1) / P;
      const double inflight = (double)grid * ring * slot_bytes;   // code bytes in flight
      const double bw_eff = std::min(bw, inflight / latency);
      const double part_bytes = S > 1 ? 8.0 * S * M * g.ntiles * kTileRows : 0.0;
      // split-K: the CTA that sums a tile reads S partials for each of its
      // 128 M (m, row) pairs, in rounds of 16 loads (~1.2 us a round).  M = 1:
      // summed per tile by the epilogue while MMAs go on (within the fixed
      // split-K tail below).  Else M x 128 / 768 pairs per thread of the whole
      // CTA after the main loop, about units / S tiles per CTA (rotated tile
      // orders).
      const bool now = M == 1;
      const int rounds = (kTileRows * M + kThreads - 1) / kThreads * ((S + 15) / 16);
      const double red = S <= 1 || now ? 0.0 : (double)((units + S - 1) / S) * rounds * 1.2e-6;
      const double tail = S > 1 ? 2.5e-6 + red : 0.0;
      const double t_cta = units * (4.0 * CB * t_mma + spu * 90.0 / clk + 300.0 / clk + (S > 1 ? t_tile : 0.0));
      const double t = std::max(t_cta, (code_bytes + part_bytes) / bw_eff) + tail;
      if (t < best_t * 0.999) {
        best_t = t;
        best.S = S; best.P = P; best.CB = CB; best.ring = ring; best.stream = stream;
        best.smem = std::max<size_t>(kSmemMin, 1024 + (size_t)b_bytes + (size_t)ring * sbytes);
      }
    }
  }
  return best;
}

// How the decode kernel would build its B operand at batch M: 2 polyphase,
// 1 dense G, 0 not at all (the scratch does not fit the free ring slots, or
// the build would take too many MMA steps per warp).
int fused_build(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  if (M < 1 || M > kMaxFuseM) return 0;
  if (g.block % 16 != 0 || g.n_b % 8 != 0 || !pl->d_g_frag) return 0;
  const DecodeConfig& dc = decode_config(pl, M);
  if (dc.S < 1) return 0;
  // MMA steps per builder warp for the widest chunk: (m, b) row tiles x code
  // tiles x 16-deep steps over B, shared by the 16 warps.
  const int64_t nbi = ((int64_t)dc.CB * kBlk + g.n_b - 1) / g.n_b + 1;
  const int64_t rt = ((int64_t)M * nbi + 15) / 16;
  const int64_t steps = rt * (g.n_b / 8) * (g.block / 16) / (kBuildThreads / 32);
  if (steps > kMaxBuildSteps) return 0;
  // the fp32 x_tilde scratch (and the polyphase build's u rows and table)
  // lives in the ring slots the first kFusePre stages do not use
  int sb = 0, nbuf = 0, dbase = 0;
  tmem_split(dc.NP, &sb, &nbuf, &dbase);
  const size_t slot = (size_t)sb * kTileRows * kBlk * g.bits / 8;
  if (dc.ring <= kFusePre) return 0;
  const size_t room = (size_t)(dc.ring - kFusePre) * slot;
  const size_t scratch = (size_t)M * dc.CB * kXtStride * sizeof(float);
  const size_t poly = (size_t)2 * 16 * rt * (g.block + 8) * sizeof(uint16_t) + (size_t)pl->poly_bytes +
                      sizeof(int) * ((size_t)g.n_b + 2 * 16 * rt);
  if (pl->d_poly && scratch + poly <= room) return 2;
  return scratch <= room ? 1 : 0;
}

}  // namespace sdq

// Host-only launch-shape query (sizing and tests; see include/sdq.h).
extern "C" int sdq_decode_launch_shape(const sdq_layer_desc* desc, int32_t M, int32_t sm_count, int64_t* out) {
  using namespace sdq;
  if (!desc || !out || M < 1 || M > kMaxDecodeM || sm_count < 1) return SDQ_ERR_INVALID_ARG;
  sdq_plan_s pl{};
  const int st = validate(desc, &pl.geo);
  if (st != SDQ_OK) return st;
  pl.desc = *desc;
  pl.sm_count = sm_count;
  const DecodeConfig dc = decode_config_search(&pl, M);
  if (dc.S < 1) return SDQ_ERR_UNSUPPORTED;
  int sb = 0, nbuf = 0, dbase = 0;
  tmem_split(dc.NP, &sb, &nbuf, &dbase);
  const int64_t blk = (int64_t)kTileRows * kBlk * pl.geo.bits / 8;
  const int64_t v[13] = {dc.T, dc.NP, dc.S, dc.P, dc.CB, dc.ring, dc.stream, (int64_t)dc.smem, sb, nbuf,
                         sb * (blk + (dc.stream ? (int64_t)dc.NP * 128 : 0)),
                         dc.stream ? 0 : (int64_t)dc.CB * dc.NP * 128, kSmemMax + 1024};
  for (int i = 0; i < 13; ++i) out[i] = v[i];
  return SDQ_OK;
}

namespace sdq {

bool decode_fusable(const sdq_plan_s* pl, int M, const uint16_t* x) {
  return (reinterpret_cast<uintptr_t>(x) & 15u) == 0 && fused_build(pl, M) != 0;
}

cudaError_t launch_decode(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st, int early, const uint16_t* x) {
  const Geometry& g = pl->geo;
  const DecodeConfig& dc = decode_config(pl, M);
  if (dc.S < 1) return cudaErrorNotSupported;   // the B operand of a k chunk does not fit
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  DecodeParams p;
  p.codes = codes; p.alpha = alpha; p.y = y;
  p.bimg = base + L.bimg;
  p.sexp = reinterpret_cast<const int*>(base + L.sexp);
  p.part = reinterpret_cast<float*>(base + L.part);
  p.cnt = reinterpret_cast<uint64_t*>(base + L.cnt);
  p.rec = reinterpret_cast<uint64_t*>(base + L.err);
  p.call = next_call_number();
  p.fused = x != nullptr;
  p.x = x; p.g_frag = pl->d_g_frag; p.gnorm = pl->gnorm;
  p.use_poly = p.fused && fused_build(pl, M) == 2;
  p.poly = pl->d_poly; p.poly_p = pl->poly_p; p.poly_q = pl->poly_q; p.poly_bytes = pl->poly_bytes;
  p.fwht = pl->desc.hadamard != 0;
  p.K = g.k_in; p.B = g.block; p.n_b = g.n_b; p.k_eff = g.k_eff;
  if (p.fused) early = 0;   // x and the codes may come from the preceding grid
  p.stream = !p.fused && dc.stream;
  if (p.stream) early = 0;  // every stage carries B rows written by the preceding grid
  p.M = M; p.T = dc.T; p.NP = dc.NP; p.S = dc.S; p.P = dc.P; p.CB = dc.CB;
  p.KB = (int)(g.k_eff_pad / kBlk); p.ring = dc.ring;
  tmem_split(dc.NP, &p.sb, &p.nbuf, &p.dbase);
  p.n_out = g.n_out; p.ntiles = g.ntiles; p.ngroups = g.ngroups; p.ternary = g.bits == 2;
  p.early = early;
  p.blk_bytes = (uint32_t)(kTileRows * kBlk * g.bits / 8);
  p.slot_bytes = p.sb * (p.blk_bytes + (p.stream ? (uint32_t)dc.NP * 128 : 0u));
  p.b_bytes = p.stream ? 0u : (uint32_t)(dc.CB * dc.NP * 128);
  static std::atomic<int> smem_set[2][64];   // per mode and device: limit raised to kSmemMax + 1 KB
  if (p.stream) {
    cudaError_t e = smem_limit_once(decode_kernel<true>, kSmemMax + 1024, pl->device, smem_set[1]);
    if (e != cudaSuccess) return e;
    return launch_pdl(decode_kernel<true>, dim3(dc.S * dc.P), dim3(kThreads), dc.smem, st, p);
  }
  cudaError_t e = smem_limit_once(decode_kernel<false>, kSmemMax + 1024, pl->device, smem_set[0]);
  if (e != cudaSuccess) return e;
  return launch_pdl(decode_kernel<false>, dim3(dc.S * dc.P), dim3(kThreads), dc.smem, st, p);
}

}  // namespace sdq
