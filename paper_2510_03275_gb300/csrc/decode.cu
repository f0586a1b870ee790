// K4: decode contraction (M <= 64) on the 5th-generation tensor cores, with
// the code operand expanded into tensor memory as 4-bit floats.
//
//   y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]        (section 3.5, eq. 12)
//
// A skinny contraction whose cost is streaming the packed codes (2 or 1 bits
// per weight sample) from HBM.  The products run on
// tcgen05.mma kind::mxf4.block_scale (M = 128, N = NP, K = 64 per
// instruction, e2m1 operands with one ue8m0 scale per 32 K) and the CUDA
// cores only expand:
//   A (TMEM)  the codes of a 128-row tile as e2m1 +-2.0 / 0, 8 per 32-bit
//             column: thread = TMEM lane = weight row, one shift and one
//             mask per 8 ternary codes (decode_stage_k order), written with
//             tcgen05.st straight from registers; 16 columns per 128 codes
//   B (smem)  the activations as T e2m1 terms per batch row m, per group g of
//             32 codes: x_tilde[m, g] = 2^e sum_t 8^-t q_t with 2^e from the
//             group's own maximum (|x_tilde 2^-e| < 4, each later term the
//             8x-scaled rounding error of the one before), N = M T rows
//             rounded up to 16, K-major, 128-byte swizzle, two 128-code
//             blocks per 128-byte row: the decode prepare kernel writes this
//             image for all of K once per call (n_b a multiple of 64) and
//             each CTA copies its k chunk's part; otherwise the CTA forms its
//             part from the prepared fp32 x_tilde
//   scales    A: 1.0 everywhere; B: 2^(e - 3t) for term row m T + t and
//             32-code group g, one set of TMEM columns per 128-code block
//             (scale id 0 for its first MMA, 2 for its second)
//   D (TMEM)  fp32, 128 lanes x NP columns
// so that y[m, r] = alpha_r / 2 * sum_t D[r, m T + t].
//
// A stage is up to sb blocks of 128 codes (2 sb MMAs): every mbarrier wait
// of an MMA-issuing thread costs about as much as several MMAs, so the CTA
// runs two independent pipelines e = 0, 1 on alternate stages (i = e mod 2),
// each with its own producer thread, two expander sets, MMA issuer, two
// TMEM slots and accumulator; the epilogue adds the two accumulators.  Set
// t of pipeline e owns TMEM slot 2e + t and expands the pipeline's stages
// j = t (mod 2): every mbarrier has one producer and one consumer that both
// walk its phases in order.
//
// CTA (k chunk s, row set p) of one SM, 24 warps:
//   warps 0, 1    lane 0 of warp e streams pipeline e's stages (one 128-row
//                 tile x up to sb * 128 codes = contiguous slabs of the tiled
//                 layout) into its shared-memory ring slots with bulk
//                 copies; warp 0 also owns the TMEM allocation
//   warps 2, 3    lane 0 of warp 2 + e issues pipeline e's MMAs, commits to
//                 the stage's TMEM slot and, after its last stage of a row
//                 tile, to its accumulator
//   warps 4..19   first the B operand and its scales, then the expanders:
//                 set x = 2e + t (warps 4 + 4x .. 7 + 4x, one per TMEM lane
//                 quadrant) expands stages i = e + 2t (mod 4) into TMEM slot x
//   warps 20..23  epilogue: read and add the accumulators, sum the terms,
//                 scale and store y; with split-K (S > 1) either add into y
//                 with float atomics (y cleared by the prepare kernel of the
//                 same call: sdq_linear_forward) or store a partial, and after
//                 the main loop take the tiles' tickets; the CTA with a tile's
//                 last ticket sums its S partials in a fixed order
//                 (deterministic: sdq_contract)
// With `early` set the producers start the code stream before waiting for
// the preceding grid (codes are never written by the prep kernels).
// Every mbarrier wait is bounded (about 2 s); a timeout writes the call's
// tag into the workspace's call record and the CTA drains its copies and
// MMAs before freeing TMEM.
#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBlk = 128;                        // codes per block (2 MMAs of K = 64)
constexpr int kAColsPerBlk = kBlk / 8;           // TMEM columns of a block's e2m1 codes
constexpr int kProducers = 2;                    // warps 0, 1
constexpr int kIssuerWarp0 = 2;                  // warps 2, 3
constexpr int kSlots = 2;                        // TMEM A slots (and expander sets) per pipeline
constexpr int kMaxSb = 4;                        // at most 4 blocks per stage
constexpr int kExpWarp0 = 4;                     // warps 4..19
constexpr int kExpSets = 2 * kSlots;
constexpr int kEpiWarp0 = kExpWarp0 + 4 * kExpSets;   // warps 20..23
constexpr int kThreads = 32 * (kEpiWarp0 + 4);   // 768
constexpr int kMaxRing = 24;
constexpr int kMaxSpu = 128;                     // stages per row tile (config search bound)
constexpr int kSmemMax = 224 * 1024;
constexpr int kSmemMin = 120 * 1024;             // > half an SM: one CTA per SM
constexpr int kBuildThreads = 32 * 4 * kExpSets; // the expander warps load the B operand
constexpr int kRedWords = 64;                    // split-K sums summed CTA-wide: first 2048 tiles
constexpr int kSfaCols = 4;                      // A scales: column 32 q + lane r holds row r's
static_assert(kMaxRing <= 32 && 2 * kSlots + 7 <= 16 && kRedWords == 64 && kMaxSpu < 160,
              "the prologue's per-warp set-up assumes these bounds");

struct DecodeParams {
  const uint32_t* codes;
  const float* alpha;
  const float* xt;       // prepared x_tilde, M x kpad fp32 (bsrc = 1)
  const uint8_t* bimg;   // prepared B operand image (bsrc = 2)
  const uint8_t* sfbw;   // prepared B scale words, KB x NP (bsrc = 2)
  float* y;              // M x n_out
  float* part;           // S x M x (ntiles * 128) split-K partials
  uint64_t* cnt;         // ntiles split-K tickets (ticket_take)
  uint64_t* rec;         // call record
  uint64_t call;         // call tag
  int bsrc;              // B operand from: 1 prepared x_tilde, 2 prepared image
  int64_t k_eff, kpad;
  int M, T, NP, S, P, CB, KB, ring, sb, nbuf, dbase, sfa, sfb, ss;
  int n_out, ntiles, ngroups, ternary, early;
  int atomic_y;          // split-K by float atomic adds into y (zeroed by the prepare kernel)
  uint32_t blk_bytes, slot_bytes, b_bytes, sfb_bytes;
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

// The B operand of the chunk from the prepared fp32 x_tilde, where the
// prepare kernel wrote no image (n_b not a multiple of 64): T e2m1 terms per
// batch row and 32-code group, and the group's term scales, as the prepare
// kernel forms them.  Task (m, block bl, g8) of one thread: the 8 MMA
// positions kap = 8 g8 .. 8 g8 + 7 of block bl (one 32-bit word of nibbles
// per term); the four tasks of a 32-position scale group are consecutive
// lanes and share their maximum by shuffles.  Each term row's word goes to
// the CTA's image (two 128-code blocks per 128-byte row, 128-byte swizzle);
// the scale bytes 2^(e - 3t) to `sfbs`, one 32-bit word per (block, term
// row): byte 2 mu + beta = scale of K group beta of the block's MMA mu.
__device__ void write_terms(const DecodeParams& p, uint8_t* bop, uint8_t* sfbs, int kb0, int ncb, int et) {
  const bool ter = p.ternary != 0;
  const int ntask = p.M * ncb * 16;
  const int64_t lim = min((int64_t)ncb * kBlk, p.k_eff - (int64_t)kb0 * kBlk);   // chunk codes below K_eff
  const int lane = et & 31;
  for (int task0 = (et >> 5) * 32; task0 < ntask; task0 += kBuildThreads) {
    const int task = task0 + lane;
    const bool act = task < ntask;
    const int m = act ? task / (ncb * 16) : 0;
    const int rem = act ? task - m * ncb * 16 : 0, bl = rem >> 4, g8 = rem & 15;
    float v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int kl = decode_stage_k(8 * g8 + i, ter);
      const int64_t loc = (int64_t)bl * kBlk + kl;
      v[i] = 0.f;
      if (act && loc < lim) v[i] = __ldcg(p.xt + (size_t)m * p.kpad + (size_t)kb0 * kBlk + loc);
    }
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) mx = fmaxf(mx, fabsf(v[i]));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    int e = -125;
    if (mx > 0.f) {   // mx < 2^E, so |v 2^-(E - 2)| < 4
      int E = 0;
      frexpf(mx, &E);
      e = E - 2;
    }
    const float inv = ldexpf(1.f, -e);
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] *= inv;
    if (!act) continue;
    const int kb = kb0 + bl;
    uint8_t* img = bop + (size_t)((kb >> 1) - (kb0 >> 1)) * p.NP * 128;
    const int chunk = 4 * (kb & 1) + (g8 >> 2), off = 4 * (g8 & 3);
    for (int t = 0; t < p.T; ++t) {
      uint32_t word = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {   // nibble 2i = v[2i], 2i + 1 = v[2i + 1]
        float2 q;
        word |= e2m1x2(v[2 * i], v[2 * i + 1], &q) << (8 * i);
        v[2 * i] = (v[2 * i] - q.x) * 8.f;
        v[2 * i + 1] = (v[2 * i + 1] - q.y) * 8.f;
      }
      const int row = m * p.T + t;
      *reinterpret_cast<uint32_t*>(img + row * 128 + ((chunk ^ (row & 7)) << 4) + off) = word;
      if ((g8 & 3) == 0) sfbs[((size_t)bl * p.NP + row) * 4 + (g8 >> 2)] = (uint8_t)max(1, min(254, 127 + e - 3 * t));
    }
  }
}

// The scale factors into TMEM, columns from sfa on: A's (1.0) in the first
// kSfaCols, then per block bl the set of ss columns of B's: term row n at
// column n / 32 of the set, lane n mod 32 of every lane quadrant (each
// quadrant of the MMA reads its own copy).  32 columns per tcgen05.st (the
// column count is rounded up to 32 in the TMEM plan); the four builder warps
// of a lane quadrant share the stores.
__device__ void store_scales(const DecodeParams& p, uint32_t tmem, const uint8_t* sfbs, int ncb, int warp, int lane) {
  const int q = warp & 3, x = (warp - kExpWarp0) >> 2;
  const uint32_t lq = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)p.sfa;
  const int ncs = (p.NP + 31) / 32, MT = p.M * p.T, ncol = kSfaCols + ncb * p.ss;
  const uint32_t* w = reinterpret_cast<const uint32_t*>(sfbs);
  for (int c0 = 32 * x; c0 < ncol; c0 += 128) {
    uint32_t v[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int cc = c0 + i - kSfaCols;
      uint32_t val = kUnitScales;
      if (cc >= 0 && cc < ncb * p.ss) {
        const int bl = cc / p.ss, j = cc - bl * p.ss, n = 32 * j + lane;
        if (j < ncs && n < MT) val = w[bl * p.NP + n];
      }
      v[i] = val;
    }
    tmem_st32(lq + (uint32_t)c0, v);
  }
}

__global__ void __launch_bounds__(kThreads, 1) decode_kernel(DecodeParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t c_full[kMaxRing], c_empty[kMaxRing];
  __shared__ __align__(8) uint64_t a_full[2 * kSlots], a_empty[2 * kSlots];
  __shared__ __align__(8) uint64_t acc_full[2][2], acc_empty[2][2], b_full, b_copy, mma_done[2];
  __shared__ uint32_t tmem_base;
  __shared__ uint32_t red_bits[kRedWords];  // tiles whose split-K sum this CTA owes (all threads sum)
  __shared__ int sblk[kMaxSpu + 1];         // first block of stage j of a tile

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int sidx = blockIdx.x % p.S, prow = blockIdx.x / p.S;
  const int kb0 = sidx * p.CB;
  const int ncb = min(p.CB, p.KB - kb0);                        // blocks of this chunk
  const int spu = max((ncb + p.sb - 1) / p.sb, min(2, ncb));   // stages per tile
  const int nunits = (p.ntiles - prow + p.P - 1) / p.P;         // row tiles of this CTA
  // The CTAs of a row set (one per k chunk) walk its tiles in rotated orders:
  // unit u is tile prow + ((u + rot) mod nunits) P.
  const int rot = (int)(((int64_t)sidx * ((nunits + p.S - 1) / p.S)) % max(nunits, 1));
  const int nstages = nunits * spu;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* bop = base;                                          // B image: b_bytes
  uint8_t* sfbs = base + p.b_bytes;                             // CB x NP B scale words: sfb_bytes
  uint8_t* ring = sfbs + p.sfb_bytes;                           // ring x slot_bytes

  // Set-up spread over warps 1.. (warp 0 allocates TMEM meanwhile).
  if (warp == 1 && lane < p.ring) {
    mbar_init(&c_full[lane], 1);
    mbar_init(&c_empty[lane], 4);   // one arrival per expander warp of the slot's set
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
      mbar_init(&b_copy, 1);
    } else if (lane == 2 * kSlots + 5 || lane == 2 * kSlots + 6) {
      mbar_init(&mma_done[lane - 2 * kSlots - 5], 1);
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
  // (the builders wait inside their build; the producers, with `early`, after
  // their first stages)
  const bool builder = warp >= kExpWarp0 && warp < kEpiWarp0;
  if (!builder && (warp >= kProducers || !p.early)) pdl_wait();
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp < kProducers) {
    if (lane == 0) {
      // Producer of pipeline `warp`: stages i = warp (mod 2), ring slots
      // i mod ring (ring is even).  Stage (unit u, j) is the slabs
      // (tile, 2 b) .. (tile, 2 b' - 1) of its blocks [b, b'), adjacent in the
      // tiled layout.
      int last_i = -1;
      int u = 0, j = warp;
      while (j >= spu) { j -= spu; ++u; }
      const uint64_t pol = l2_policy_evict_first();   // codes are read once per call
      for (int i = warp; i < nstages && ok; i += kProducers) {
        const int slot = i % p.ring, r = i / p.ring;
        if (r > 0) ok = mbar_wait(&c_empty[slot], (r - 1) & 1);
        if (!ok) break;
        const int b0 = sblk[j], b1 = sblk[j + 1];
        const int tile = prow + (u + rot < nunits ? u + rot : u + rot - nunits) * p.P;
        const uint8_t* src = reinterpret_cast<const uint8_t*>(p.codes) +
                             ((size_t)tile * p.KB + kb0 + b0) * p.blk_bytes;
        const uint32_t bytes = (uint32_t)(b1 - b0) * p.blk_bytes;
        mbar_expect_tx(&c_full[slot], bytes);
        bulk_g2s_hint(ring + (size_t)slot * p.slot_bytes, src, bytes, &c_full[slot], pol);
        last_i = i;
        j += kProducers;
        while (j >= spu) { j -= spu; ++u; }
      }
      if (p.early) pdl_wait();
      // Every copy this thread issued has landed before the CTA may exit.
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
      const uint32_t idesc0 = mxf4_idesc(p.NP), idesc1 = idesc0 | (2u << 4);   // B scale bytes 0-1 / 2-3
      // Per stage: one wait, 2 nb MMAs, one commit; stage bookkeeping is
      // kept incremental (a single thread's scalar latency is on the path).
      const uint64_t bd0 = sw128_desc(sbase);
      const uint64_t astep = (uint64_t)((p.NP * 128) >> 4);   // descriptor units per image row pair
      const uint32_t sfa = tmem + (uint32_t)p.sfa, sfb0 = tmem + (uint32_t)p.sfb;
      const uint32_t aslot = (uint32_t)(kAColsPerBlk * p.sb);
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
        uint32_t at = tmem + (uint32_t)a * aslot;
        for (int bb = 0; bb < nb; ++bb, at += kAColsPerBlk) {
          const int bl = b0 + bb, kb = kb0 + bl;
          const uint64_t bd = bd0 + (uint64_t)((kb >> 1) - (kb0 >> 1)) * astep + 4u * (uint32_t)(kb & 1);
          const uint32_t sfb = sfb0 + (uint32_t)(bl * p.ss);
          umma_mxf4_ts(dt, at, bd, idesc0, sfa, sfb, (first && bb == 0) ? 0u : 1u);
          umma_mxf4_ts(dt, at + 8, bd + 2, idesc1, sfa, sfb, 1u);
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
    // ------------------------------------------------ builders, then expanders
    const int et = tid - 32 * kExpWarp0;
    if (p.bsrc == 2) {
      // the prepared image rows of the chunk's blocks and their scale words
      pdl_wait();
      if (et == 0) {
        const int a0 = kb0 >> 1, a1 = (kb0 + ncb - 1) >> 1;
        const uint32_t ib = (uint32_t)(a1 - a0 + 1) * p.NP * 128, sb = (uint32_t)ncb * p.NP * 4;
        mbar_expect_tx(&b_copy, ib + sb);
        bulk_g2s(bop, p.bimg + (size_t)a0 * p.NP * 128, ib, &b_copy);
        bulk_g2s(sfbs, p.sfbw + (size_t)kb0 * p.NP * 4, sb, &b_copy);
      }
      ok = mbar_wait(&b_copy, 0);
      if (!ok) mbar_wait(&b_copy, 0);   // a copy still in flight must land before the CTA exits
    } else {
      pdl_wait();
      write_terms(p, bop, sfbs, kb0, ncb, et);
      fence_proxy_async_smem();   // generic-proxy stores -> the MMAs' async-proxy reads
    }
    named_bar_sync(3, kBuildThreads);
    store_scales(p, tmem, sfbs, ncb, warp, lane);
    tmem_st_wait();
    tc_fence_before();
    named_bar_sync(3, kBuildThreads);
    if (et == 0) mbar_arrive(&b_full);

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
          // e2m1 nibble [sign, code bit 0, 0, 0]: +-2.0 or 0 (decode_stage_k order)
          uint32_t v[16];
          if (p.ternary) {
#pragma unroll
            for (int wi = 0; wi < 8; ++wi) {
              v[2 * wi] = (w[bb][wi] << 2) & 0xCCCCCCCCu;   // even codes
              v[2 * wi + 1] = w[bb][wi] & 0xCCCCCCCCu;      // odd codes
            }
          } else {   // words hold the inverted bits: 1 = -1
#pragma unroll
            for (int wi = 0; wi < 4; ++wi)
#pragma unroll
              for (int k = 0; k < 4; ++k) v[4 * wi + k] = ((w[bb][wi] << (3 - k)) & 0x88888888u) | 0x44444444u;
          }
          tmem_st16(lane_addr + (uint32_t)(a * kAColsPerBlk * p.sb + kAColsPerBlk * bb), v);
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
    call_record_start(p.rec, p.call, blockIdx.x == 0 && et == 0);
    // the k-chunk-0 CTA of each row set puts this call's tag into the row
    // set's tickets while the main loop runs
    if (p.S > 1 && !p.atomic_y && sidx == 0 && et < 32)
      for (int u = et; u < nunits; u += 32) ticket_install(p.cnt + prow + u * p.P, p.call);
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
      float acc = 0.f;
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
            acc += (in0 ? __uint_as_float(r0[i]) : 0.f) + (in1 ? __uint_as_float(r1[i]) : 0.f);
            if (++t == p.T) {   // the terms of batch row m, already scaled by their B scales
              if (p.S == 1) {
                if (live) p.y[(size_t)m * p.n_out + row] = sa * acc;
              } else if (p.atomic_y) {
                if (live) atomicAdd(p.y + (size_t)m * p.n_out + row, sa * acc);
              } else {
                p.part[((size_t)sidx * p.M + m) * NR + row] = acc;
              }
              acc = 0.f; t = 0; ++m;
            }
          }
        }
      }
      kc[0] += in0;
      kc[1] += in1;
    }
  }
  if (!ok) call_record_fail(p.rec, p.call);
  tc_fence_before();
  const bool cta_ok = __syncthreads_and(ok ? 1 : 0) != 0;
  // Split-K, after the main loop: one thread per row tile of this CTA takes
  // the tile's ticket (after the barrier above, which orders every thread's
  // partial stores before the ticket's release fence).  Per-tile tickets
  // while the next tiles' MMAs run cost each tile a fence and an atomic round
  // trip in the epilogue, which then held up the MMAs.  Then every thread of
  // the CTA sums the S partials of the tiles whose last ticket it took, in
  // k-chunk order (deterministic): (m, row) pairs, consecutive threads on
  // consecutive rows, 16 loads in flight.
  if (p.S > 1 && !p.atomic_y && cta_ok) {   // (uniform: the barrier below)
    const int NR = p.ntiles * kTileRows;
    const size_t sstride = (size_t)p.M * NR;
    auto sum_pair = [&](int row, int mm) {
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
    };
    for (int u = tid; u < nunits; u += kThreads) {
      const int ut = u + rot < nunits ? u + rot : u + rot - nunits;
      const uint32_t n = ticket_take(p.cnt + prow + ut * p.P, p.call, (uint32_t)p.S);
      if (n == 0) call_record_fail(p.rec, p.call);
      if (n == (uint32_t)p.S) {
        if (ut < 32 * kRedWords) {
          atomicOr(&red_bits[ut >> 5], 1u << (ut & 31));
        } else {   // beyond the bit set (more than 2048 row tiles per CTA): this thread alone
          const int row0 = (prow + ut * p.P) * kTileRows;
          for (int i = 0; i < kTileRows * p.M; ++i) {
            const int mm = i / kTileRows, row = row0 + (i - mm * kTileRows);
            if (row < p.n_out) sum_pair(row, mm);
          }
        }
      }
    }
    __syncthreads();
    for (int w = 0; w < kRedWords; ++w) {
      uint32_t bits = red_bits[w];
      while (bits) {
        const int u = 32 * w + __ffs(bits) - 1;
        bits &= bits - 1;
        const int row0 = (prow + u * p.P) * kTileRows;
        for (int i = tid; i < kTileRows * p.M; i += kThreads) {
          const int mm = i / kTileRows, row = row0 + (i - mm * kTileRows);
          if (row < p.n_out) sum_pair(row, mm);
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

}  // namespace

// Launch shape for batch M: the (S, P) grid of at most one CTA per SM (more
// only where nothing else fits) that minimises a simple time model: the larger of the MMA time of the busiest
// CTA and the HBM time of codes plus split-K partials (the bytes in flight
// capped by the CTAs' code rings), plus the split-K tail (one fence, one
// ticket, the final sums).  TMEM holds, from column 0: four A slots of sb
// blocks (16 sb columns each), the A scales (4 columns), one set of
// ss = 4 ceil(ceil(NP / 32) / 4) B scale columns per block of the chunk, and
// at the top the accumulators (2 pipelines x nbuf x NP columns).
DecodeConfig decode_config_search(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  DecodeConfig best{};
  best.M = M;
  best.T = decode_terms(M);
  best.NP = (M * best.T + 15) / 16 * 16;
  best.nbuf = best.NP <= 64 ? 2 : 1;
  best.dbase = 512 - 2 * best.nbuf * best.NP;
  best.ss = 4 * (((best.NP + 31) / 32 + 3) / 4);
  const int KB = (int)(g.k_eff_pad / kBlk);
  const int sms = std::max(1, pl->sm_count);
  const int blk_bytes = kTileRows * kBlk * g.bits / 8;
  // M = 1 constants fitted to measured launches: each split-K tile costs
  // its epilogue (partial stores, a release fence and a ticket round trip
  // while the code stream loads HBM) beyond its MMAs, and the ring's copies
  // see a longer loaded latency.
  const double clk = 1.9e9, bw = 6.5e12;
  const double latency = M == 1 ? 3.0e-6 : 2.2e-6;             // loaded HBM latency
  const double t_tile = M == 1 ? 0.5e-6 : 0.0;                 // per split-K tile
  const double t_blk = 2.0 * std::max(32.0, best.NP * 0.3) / clk;   // two MMAs, two issuers
  const double code_bytes = (double)g.ntiles * kTileRows * g.k_eff_pad * g.bits / 8;
  double best_t = 1e30;
  // k chunks beyond the SM count (CTAs in several waves) only where the
  // chunk's B operand and scales would not fit otherwise (large batches on
  // small parts)
  for (int S = 1; S <= KB && (S <= sms || best.S == 0); ++S) {
    const int CB = (KB + S - 1) / S;
    if ((S - 1) * CB >= KB) continue;                      // no empty chunk
    const int sfcols = (kSfaCols + CB * best.ss + 31) / 32 * 32;   // scale columns, stored 32 at a time
    const int sb = std::min(kMaxSb, (best.dbase - sfcols) / 64);
    if (sb < 1) continue;                                  // TMEM
    const int b_bytes = (CB / 2 + 1) * best.NP * 128;       // image rows of the chunk's blocks
    const int sfb_bytes = (CB * best.NP * 4 + 15) / 16 * 16;  // its B scale words
    const int slot_bytes = sb * blk_bytes;
    int ring = std::min(kMaxRing, (kSmemMax - 2048 - b_bytes - sfb_bytes) / slot_bytes);
    ring -= ring % kExpSets;          // each ring slot belongs to one expander set
    if (ring < kExpSets) continue;
    const int spu = std::max((CB + sb - 1) / sb, std::min(2, CB));
    if (spu > kMaxSpu) continue;
    // the B operand of the chunk, built before the first MMA: a latency
    // floor plus the e2m1 terms of CB 128-code blocks per batch row
    const double t_build = 2.0e-6 + CB * M * best.T * 4.0e-9;
    for (int P = 1; P <= std::min(g.ntiles, std::max(1, sms / S)); ++P) {
      const int grid = S * P;
      const int waves = (grid + sms - 1) / sms;
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
      const double t_cta = units * (CB * t_blk + spu * 90.0 / clk + 300.0 / clk + (S > 1 ? t_tile : 0.0));
      const double t = std::max(waves * t_cta, (code_bytes + part_bytes) / bw_eff) + tail + t_build;
      if (t < best_t * 0.999) {
        best_t = t;
        best.S = S; best.P = P; best.CB = CB; best.ring = ring; best.sb = sb;
        best.smem = std::max<size_t>(kSmemMin, 1024 + (size_t)b_bytes + sfb_bytes + (size_t)ring * slot_bytes);
      }
    }
  }
  best.sfa = 64 * best.sb;
  best.sfb = best.sfa + kSfaCols;
  return best;
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
  const int64_t blk = (int64_t)kTileRows * kBlk * pl.geo.bits / 8;
  const int64_t v[13] = {dc.T, dc.NP, dc.S, dc.P, dc.CB, dc.ring, dc.sb, dc.nbuf, (int64_t)dc.smem,
                         dc.sb * blk, (int64_t)(dc.CB / 2 + 1) * dc.NP * 128, dc.ss, kSmemMax + 1024};
  for (int i = 0; i < 13; ++i) out[i] = v[i];
  return SDQ_OK;
}

namespace sdq {

bool decode_image(const sdq_plan_s* pl) { return pl->geo.n_b % 64 == 0; }


cudaError_t launch_decode(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st, int early, int y_zeroed) {
  const Geometry& g = pl->geo;
  const DecodeConfig& dc = decode_config(pl, M);
  if (dc.S < 1) return cudaErrorNotSupported;   // no launch shape fits
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  DecodeParams p;
  p.codes = codes; p.alpha = alpha; p.y = y;
  p.xt = reinterpret_cast<const float*>(base + L.xt);
  p.bimg = base + L.bimg;
  p.sfbw = base + L.sfbw;
  p.part = reinterpret_cast<float*>(base + L.part);
  p.cnt = reinterpret_cast<uint64_t*>(base + L.cnt);
  p.rec = reinterpret_cast<uint64_t*>(base + L.err);
  p.call = call_tag(next_call_number());
  p.bsrc = decode_image(pl) ? 2 : 1;
  p.k_eff = g.k_eff; p.kpad = g.k_eff_pad;
  p.M = M; p.T = dc.T; p.NP = dc.NP; p.S = dc.S; p.P = dc.P; p.CB = dc.CB;
  p.KB = (int)(g.k_eff_pad / kBlk); p.ring = dc.ring;
  p.sb = dc.sb; p.nbuf = dc.nbuf; p.dbase = dc.dbase; p.sfa = dc.sfa; p.sfb = dc.sfb; p.ss = dc.ss;
  p.n_out = g.n_out; p.ntiles = g.ntiles; p.ngroups = g.ngroups; p.ternary = g.bits == 2;
  p.early = early;
  p.atomic_y = y_zeroed && dc.S > 1;
  p.blk_bytes = (uint32_t)(kTileRows * kBlk * g.bits / 8);
  p.slot_bytes = p.sb * p.blk_bytes;
  p.b_bytes = (uint32_t)((dc.CB / 2 + 1) * dc.NP * 128);
  p.sfb_bytes = (uint32_t)((dc.CB * dc.NP * 4 + 15) / 16 * 16);
  static std::atomic<int> smem_set[64];   // per device: limit raised to kSmemMax + 1 KB
  cudaError_t e = smem_limit_once(decode_kernel, kSmemMax + 1024, pl->device, smem_set);
  if (e != cudaSuccess) return e;
  return launch_pdl(decode_kernel, dim3(dc.S * dc.P), dim3(kThreads), dc.smem, st, p);
}

}  // namespace sdq
