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
//             N = M*T rows rounded up to 16, K-major, 128-byte swizzle,
//             written for all of K by the decode prepare kernel; each CTA
//             copies the part of its k chunk once
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
//                 layout) into its shared-memory ring slots with bulk copies;
//                 warp 0 also owns the TMEM allocation and copies the chunk's
//                 B operand
//   warps 2, 3    lane 0 of warp 2 + e issues pipeline e's MMAs, commits to
//                 the stage's TMEM slot and, after its last stage of a row
//                 tile, to its accumulator
//   warps 4..19   expanders: set x = 2e + t (warps 4 + 4x .. 7 + 4x, one per
//                 TMEM lane quadrant) expands stages i = e + 2t (mod 4) into
//                 TMEM slot x
//   warps 20..23  epilogue: read and add the accumulators, combine the
//                 terms, scale and store y, or store a split-K partial; after
//                 the CTA's last tile, one fence and one ticket per tile, and
//                 the last CTA of each tile sums its S partials in a fixed
//                 order (deterministic)
// With `early` set the producers start the code stream before waiting for
// the preceding grid (codes are never written by the prep kernels).
// Every mbarrier wait is bounded (about 2 s); a timeout sets the workspace
// error word and the CTA drains its copies and MMAs before freeing TMEM.
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

struct DecodeParams {
  const uint32_t* codes;
  const float* alpha;
  const uint8_t* bimg;   // B operand image: KB x NP x 128 bytes
  const int* sexp;       // per-batch-row scale exponents e_m
  float* y;              // M x n_out
  float* part;           // S x M x (ntiles * 128) split-K partials
  uint32_t* cnt;         // ntiles tickets (zeroed by the prep kernel)
  uint32_t* err;
  int M, T, NP, S, P, CB, KB, ring, sb, nbuf, dbase;
  int n_out, ntiles, ngroups, ternary, early;
  uint32_t blk_bytes, slot_bytes, b_bytes;
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

__global__ void __launch_bounds__(kThreads, 1) decode_kernel(DecodeParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t c_full[kMaxRing], c_empty[kMaxRing];
  __shared__ __align__(8) uint64_t a_full[2 * kSlots], a_empty[2 * kSlots];
  __shared__ __align__(8) uint64_t acc_full[2][2], acc_empty[2][2], b_full, mma_done[2];
  __shared__ uint32_t tmem_base;
  __shared__ int last[128];
  __shared__ float scale_s[kMaxDecodeM];   // 2^e_m
  __shared__ int sblk[kMaxSpu + 1];         // first block of stage j of a tile

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int sidx = blockIdx.x % p.S, prow = blockIdx.x / p.S;
  const int kb0 = sidx * p.CB;
  const int ncb = min(p.CB, p.KB - kb0);                        // blocks of this chunk
  const int spu = max((ncb + p.sb - 1) / p.sb, min(2, ncb));   // stages per tile
  const int nunits = (p.ntiles - prow + p.P - 1) / p.P;         // row tiles of this CTA
  const int nstages = nunits * spu;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* bop = base;                                          // ncb x NP x 128 bytes
  uint8_t* ring = base + p.b_bytes;                             // ring x slot_bytes

  if (tid == 0) {
    for (int i = 0; i < p.ring; ++i) {
      mbar_init(&c_full[i], 1);
      mbar_init(&c_empty[i], 4);     // one arrival per expander warp
    }
    for (int i = 0; i < 2 * kSlots; ++i) {
      mbar_init(&a_full[i], 4);
      mbar_init(&a_empty[i], 1);
    }
    for (int e = 0; e < 2; ++e)
      for (int b = 0; b < 2; ++b) {
        mbar_init(&acc_full[e][b], 1);
        mbar_init(&acc_empty[e][b], 128);
      }
    for (int j = 0; j <= spu; ++j) sblk[j] = stage_block(j, ncb, spu);
    mbar_init(&b_full, 1);
    mbar_init(&mma_done[0], 1);
    mbar_init(&mma_done[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    __syncwarp();
    tmem_alloc(&tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_launch_dependents();
  if (warp >= kProducers || !p.early) pdl_wait();
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
      bool b_loaded = warp != 0;
      const int pre = p.early ? min(2 * kProducers, nstages) : 0;
      int u = 0, j = warp;
      while (j >= spu) { j -= spu; ++u; }
      for (int i = warp; i < nstages && ok; i += kProducers) {
        if (!b_loaded && i >= pre) {
          if (p.early) pdl_wait();
          mbar_expect_tx(&b_full, p.b_bytes);
          bulk_g2s(bop, p.bimg + (size_t)kb0 * p.NP * 128, p.b_bytes, &b_full);
          b_loaded = true;
        }
        const int slot = i % p.ring, r = i / p.ring;
        if (r > 0) ok = mbar_wait(&c_empty[slot], (r - 1) & 1);
        if (!ok) break;
        const int b0 = sblk[j], b1 = sblk[j + 1];
        const int tile = prow + u * p.P;
        const uint8_t* src = reinterpret_cast<const uint8_t*>(p.codes) +
                             ((size_t)tile * p.KB + kb0 + b0) * p.blk_bytes;
        const uint32_t bytes = (uint32_t)(b1 - b0) * p.blk_bytes;
        mbar_expect_tx(&c_full[slot], bytes);
        bulk_g2s(ring + (size_t)slot * p.slot_bytes, src, bytes, &c_full[slot]);
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
      if (warp == 0 && b_loaded && !mbar_wait(&b_full, 0)) ok = false;
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
        uint64_t bd = bd0 + (uint64_t)b0 * bstep;
        uint32_t at = abase + (uint32_t)(jj & 1) * aslot;
        for (int bb = 0; bb < nb; ++bb, at += 32, bd += bstep) {
          umma_f8_ts(dt, at, bd, idesc, (first && bb == 0) ? 0u : 1u);
          umma_f8_ts(dt, at + 8, bd + 2, idesc, 1u);
          umma_f8_ts(dt, at + 16, bd + 4, idesc, 1u);
          umma_f8_ts(dt, at + 24, bd + 6, idesc, 1u);
        }
        umma_commit(&a_empty[a]);
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
    }
  } else if (warp < kEpiWarp0) {
    // ------------------------------------------------------------ expanders
    // Set x = 2e + t expands stages i = e + 2t (mod 4) in order: TMEM slot
    // x, ring slots i mod ring (ring is a multiple of 4).
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
    if (et < p.M) scale_s[et] = ldexpf(1.f, p.sexp[et]);
    named_bar_sync(2, 128);
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
      const int row = (prow + u * p.P) * kTileRows + r;
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
    }
    if (p.S > 1 && ok) {
      // Split-K: one fence for all of this CTA's partials, then one ticket
      // per tile; the CTA that takes the last ticket of a tile sums its S
      // partials in k-chunk order.
      __threadfence();
      named_bar_sync(2, 128);
      for (int u0 = 0; u0 < nunits; u0 += 128) {
        const int u = u0 + et;
        last[et] = u < nunits && atomicAdd(p.cnt + prow + u * p.P, 1u) == (uint32_t)(p.S - 1);
        named_bar_sync(2, 128);
        __threadfence();
        for (int uu = 0; uu < min(128, nunits - u0); ++uu) {
          if (!last[uu]) continue;
          const int row = (prow + (u0 + uu) * p.P) * kTileRows + r;
          if (row >= p.n_out) continue;
          const float sa = 0.5f * __ldg(p.alpha + row);
          const size_t sstride = (size_t)p.M * NR;
          for (int mm = 0; mm < p.M; ++mm) {
            const float* pr = p.part + (size_t)mm * NR + row;
            float s0 = 0.f;
            int kk = 0;
            for (; kk + 4 <= p.S; kk += 4) {
              const float a0 = __ldcg(pr + (size_t)kk * sstride), a1 = __ldcg(pr + (size_t)(kk + 1) * sstride);
              const float a2 = __ldcg(pr + (size_t)(kk + 2) * sstride), a3 = __ldcg(pr + (size_t)(kk + 3) * sstride);
              s0 = (((s0 + a0) + a1) + a2) + a3;
            }
            for (; kk < p.S; ++kk) s0 += __ldcg(pr + (size_t)kk * sstride);
            p.y[(size_t)mm * p.n_out + row] = sa * s0;
          }
        }
        named_bar_sync(2, 128);
      }
    }
  }
  if (!ok) atomicExch(p.err, 1u);
  tc_fence_before();
  __syncthreads();
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
  const double clk = 1.9e9, bw = 6.5e12, latency = 2.2e-6;   // loaded HBM latency
  const double t_mma = std::max(38.0, best.NP * 0.4) / clk;     // per MMA, two issuers
  const double code_bytes = (double)g.ntiles * kTileRows * g.k_eff_pad * g.bits / 8;
  double best_t = 1e30;
  for (int S = 1; S <= std::min(KB, sms); ++S) {
    const int CB = (KB + S - 1) / S;
    if ((S - 1) * CB >= KB) continue;                      // no empty chunk
    const int b_bytes = CB * best.NP * 128;
    int ring = std::min(kMaxRing, (kSmemMax - 2048 - b_bytes) / slot_bytes);
    ring -= ring % kExpSets;          // each ring slot belongs to one expander set
    if (ring < kExpSets) continue;
    const int spu = std::max((CB + sb - 1) / sb, std::min(2, CB));
    if (spu > kMaxSpu) continue;
    for (int P = 1; P <= std::min(g.ntiles, sms / S); ++P) {
      const int grid = S * P;
      const int units = (g.ntiles + P - 1) / P;
      const double inflight = (double)grid * ring * slot_bytes;
      const double bw_eff = std::min(bw, inflight / latency);
      const double part_bytes = S > 1 ? 8.0 * S * M * g.ntiles * kTileRows : 0.0;
      const double tail = S > 1 ? 2.5e-6 + (double)M * S * kTileRows * 4 / 40e9 : 0.0;
      const double t_cta = units * (4.0 * CB * t_mma + spu * 90.0 / clk + 300.0 / clk);
      const double t = std::max(t_cta, (code_bytes + part_bytes) / bw_eff) + tail;
      if (t < best_t * 0.999) {
        best_t = t;
        best.S = S; best.P = P; best.CB = CB; best.ring = ring;
        best.smem = std::max<size_t>(kSmemMin, 1024 + (size_t)b_bytes + (size_t)ring * slot_bytes);
      }
    }
  }
  return best;
}

cudaError_t launch_decode(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st, int early) {
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
  p.cnt = reinterpret_cast<uint32_t*>(base + L.cnt);
  p.err = reinterpret_cast<uint32_t*>(base + L.err);
  p.M = M; p.T = dc.T; p.NP = dc.NP; p.S = dc.S; p.P = dc.P; p.CB = dc.CB;
  p.KB = (int)(g.k_eff_pad / kBlk); p.ring = dc.ring;
  tmem_split(dc.NP, &p.sb, &p.nbuf, &p.dbase);
  p.n_out = g.n_out; p.ntiles = g.ntiles; p.ngroups = g.ngroups; p.ternary = g.bits == 2;
  p.early = early;
  p.blk_bytes = (uint32_t)(kTileRows * kBlk * g.bits / 8);
  p.slot_bytes = p.sb * p.blk_bytes;
  p.b_bytes = (uint32_t)(dc.CB * dc.NP * 128);
  cudaError_t e = cudaFuncSetAttribute(decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)dc.smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(decode_kernel, dim3(dc.S * dc.P), dim3(kThreads), dc.smem, st, p);
}

}  // namespace sdq
