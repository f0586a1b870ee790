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
//             32-code group g, one set of TMEM columns per 128-code block of
//             a stage, written by the expanders beside the stage's codes
//             (scale id 0 for its first MMA, 2 for its second)
//   D (TMEM)  fp32, 128 lanes x NP columns
// so that y[m, r] = alpha_r / 2 * sum_t D[r, m T + t].
//
// Issuing one of these MMAs occupies the issuing thread for about 130 cycles
// whatever N is, while MMAs issued from different warps proceed side by
// side; so the stages (sb <= 4 blocks of 128 codes each, 2 sb MMAs: large
// stages, since every stage costs each thread it passes through a few
// hundred cycles of waits and signals) of a row tile
// are dealt round-robin to `npipe` (1, 2 or 4) MMA pipelines, each with its
// own issuing warp and accumulator, and the epilogue adds the pipelines'
// accumulators.  Stage i of the CTA uses
//   ring slot i mod ring      (codes in shared memory; ring a multiple of 4)
//   producer i mod 4          (one thread issuing its bulk copies)
//   expander set i mod 4      (4 warps, one per TMEM lane quadrant)
//   TMEM A slot i mod ns      (ns = 4 or 8 slots of 16 sb columns: with 4,
//                             each expander set refills its one slot once
//                             the MMAs of its previous stage are done, the
//                             codes already in registers)
//   pipeline i mod npipe
// so that every mbarrier has one producer and one consumer that both walk its
// phases in order.
//
// CTA (k chunk s, row set p) of one SM, 28 warps:
//   warps 0..3    lane 0 of warp e issues pipeline e's MMAs (e < npipe),
//                 commits to the stage's TMEM slot and, after its last stage
//                 of a row tile, to its accumulator; warp 0 also owns the
//                 TMEM allocation
//   warps 4..7    epilogue: read and add the pipelines' accumulators, sum the
//                 terms, scale and store y; with split-K (S > 1) either add
//                 into y with float atomics (y cleared by the prepare kernel
//                 of the same call: sdq_linear_forward) or store a partial,
//                 and after the main loop take the tiles' tickets; the CTA
//                 with a tile's last ticket sums its S partials in a fixed
//                 order (deterministic: sdq_contract)
//   warps 8..23   first the B operand and its scales, then the expanders:
//                 set x (warps 8 + 4x .. 11 + 4x) expands stages i = x mod 4
//   warps 24..27  lane 0 of warp 24 + x streams stages i = x mod 4 (one
//                 128-row tile x sb * 128 codes = contiguous slabs of the
//                 tiled layout) into the ring with bulk copies: a thread
//                 starts a bulk copy only every ~600 cycles, four side by
//                 side keep an SM's share of HBM busy
// With `early` set the producers start the code stream (one stage each)
// before waiting for the preceding grid (codes are never written by the
// prep kernels), except with bstream, where each stage also copies B rows
// and scale words that grid writes.
//
// bstream (batches whose term rows make a chunk-resident B image bound the k
// chunk): each stage's image pairs and scale words are bulk-copied into its
// ring slot beside the codes, the MMA reads the stage's B rows there, and
// the stage's MMAs (not the expanders) release the slot; the k chunk is then
// free of shared-memory limits (S of 2 instead of 10-38 at M = 64, so far
// fewer split-K partial sums per output).
// Every mbarrier wait is bounded (about 2 s); a timeout writes the call's
// tag into the workspace's call record and the CTA drains its copies and
// MMAs before freeing TMEM.
#include <algorithm>
#include <cmath>
#include <type_traits>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBlk = 128;                        // codes per block (2 MMAs of K = 64)
constexpr int kAColsPerBlk = kBlk / 8;           // TMEM columns of a block's e2m1 codes
constexpr int kASlots = 8;                       // TMEM A slots at most: stage i -> slot i mod ns (4 or 8)
constexpr int kExpSets = 4;                      // expander sets: stage i -> set i mod 4
constexpr int kMaxPipes = 4;                     // MMA pipelines: stage i -> i mod npipe
constexpr int kMaxSb = 4;                        // blocks per stage (ns slots x 16 sb columns)
constexpr int kEpiWarp0 = kMaxPipes;             // warps 4..7
constexpr int kExpWarp0 = kEpiWarp0 + 4;         // warps 8..23
constexpr int kProducerWarp0 = kExpWarp0 + 4 * kExpSets; // warps 24..27
constexpr int kThreads = 32 * (kProducerWarp0 + kExpSets); // 896
constexpr int kMaxRing = 32;
constexpr int kMaxSpu = 128;                     // stages per row tile (config search bound)
constexpr int kSmemMax = 222 * 1024;
constexpr int kSmemMin = 120 * 1024;             // > half an SM: one CTA per SM
constexpr int kBuildThreads = 32 * 4 * kExpSets; // the expander warps load the B operand
constexpr int kRedWords = 64;                    // split-K sums summed CTA-wide: first 2048 tiles
constexpr int kSfaCols = 4;                      // A scales: column 32 q + lane r holds row r's
constexpr int kAlphaAhead = 4;                   // epilogue: alpha loads this many row tiles ahead
constexpr int kRingBytes = 160 * 1024;           // code bytes in flight per CTA (target)
constexpr int kEarlyStages = 1;                  // stages per producer issued before the preceding grid completes
static_assert(kMaxRing <= 32 && kASlots == 8 && 2 * kMaxPipes + 1 + kMaxPipes <= 32 && kRedWords == 64 &&
                  kMaxSpu < 160 && kMaxRing % kExpSets == 0,
              "the prologue's per-warp set-up and the stage maps assume these bounds");

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
  int M, T, NP, S, P, CB, KB, ring, sb, nbuf, npipe, ns, ns_log2, dbase, sfa, sfs, ss, sss;
  int n_out, ntiles, ngroups, ternary, early;
  int atomic_y;          // add into y with float reductions (y zeroed by the prepare kernel, or y += result)
  uint32_t blk_bytes, slot_bytes, b_bytes, sfb_bytes;
  int brow;   // image rows per block pair in shared memory (8 or NP)
  int bstream;          // stage B rows and scale words stream into the ring slot
  uint32_t boff, soff;  // their offsets in the slot (bstream)
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
__device__ __noinline__ void write_terms(const DecodeParams& p, uint8_t* bop, uint8_t* sfbs, int kb0, int ncb, int et) {
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

// n 16-byte words global -> shared by the kBuildThreads builder threads as
// cp.async copies, all in flight at once (completion: cp_async_wait_all).
__device__ __forceinline__ void copy_lsu(uint4* dst, const uint4* src, int n, int et) {
  for (int t = et; t < n; t += kBuildThreads) cp_async16(dst + t, src + t, 16);
}

// kTernary: 2-bit ternary codes, else 1-bit binary (one instantiation each,
// so that the expander's loop carries only its own code path).
template <bool kTernary>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(DecodeParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t c_full[kMaxRing], c_empty[kMaxRing];
  __shared__ __align__(8) uint64_t a_full[kASlots], a_empty[kASlots];
  __shared__ __align__(8) uint64_t acc_full[kMaxPipes][2], acc_empty[kMaxPipes][2], b_full;
  __shared__ __align__(8) uint64_t mma_done[kMaxPipes];
  __shared__ uint32_t tmem_base;
  __shared__ uint32_t red_bits[kRedWords];  // tiles whose split-K sum this CTA owes (all threads sum)
  __shared__ int sblk[kMaxSpu + 1];         // first block of stage j of a tile
  __shared__ float s_alpha[kAlphaAhead][kTileRows];   // epilogue: alpha of the next row tiles

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int sidx = blockIdx.x % p.S, prow = blockIdx.x / p.S;
  const int kb0 = sidx * p.CB;
  const int ncb = min(p.CB, p.KB - kb0);                        // blocks of this chunk
  // stages per tile; with bstream whole block pairs per stage (the image
  // interleaves a pair's two blocks in its 128-byte rows)
  const int npairs = (ncb + 1) >> 1;
  const int spu = p.bstream ? max((2 * npairs + p.sb - 1) / p.sb, min(2, npairs))
                            : max((ncb + p.sb - 1) / p.sb, min(2, ncb));
  const int nunits = (p.ntiles - prow + p.P - 1) / p.P;         // row tiles of this CTA
  // The CTAs of a row set (one per k chunk) walk its tiles in rotated orders:
  // unit u is tile prow + ((u + rot) mod nunits) P.
  const int rot = (int)(((int64_t)sidx * ((nunits + p.S - 1) / p.S)) % max(nunits, 1));
  const int nstages = nunits * spu;
  const int np = p.npipe;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* bop = base;                                          // B image: b_bytes
  uint8_t* sfbs = base + p.b_bytes;                             // CB x NP B scale words: sfb_bytes
  uint8_t* ring = sfbs + p.sfb_bytes;                           // ring x slot_bytes

  // Set-up spread over warps 1.. (warp 0 allocates TMEM meanwhile).
  if (warp == 1) {
    if (lane < p.ring) {
      mbar_init(&c_full[lane], 1);
      // one arrival per expander warp of the slot's set, or (bstream: the
      // MMAs read the slot's B rows) the commit of the stage's MMAs
      mbar_init(&c_empty[lane], p.bstream ? 1 : 4);
    }
  } else if (warp == 2) {
    if (lane < kASlots) {
      mbar_init(&a_full[lane], 4);
      mbar_init(&a_empty[lane], 1);
    }
  } else if (warp == 3) {
    if (lane < 2 * kMaxPipes) {
      mbar_init(&acc_full[lane >> 1][lane & 1], 1);
      mbar_init(&acc_empty[lane >> 1][lane & 1], 128);
    } else if (lane == 2 * kMaxPipes) {
      mbar_init(&b_full, 1);
    } else if (lane < 2 * kMaxPipes + 1 + kMaxPipes) {
      mbar_init(&mma_done[lane - 2 * kMaxPipes - 1], 1);
    }
  } else if (warp >= kExpWarp0 && warp < kExpWarp0 + (kMaxSpu + 32) / 32) {
    const int j = tid - 32 * kExpWarp0;
    if (j <= spu) sblk[j] = p.bstream ? min(ncb, 2 * stage_block(j, npairs, spu)) : stage_block(j, ncb, spu);
  } else if (warp >= kExpWarp0 + 6 && warp < kExpWarp0 + 8) {
    red_bits[tid - 32 * (kExpWarp0 + 6)] = 0u;
  }
  if (warp >= 1 && warp <= 3) fence_mbar_init();
  if (warp == 0) {
    __syncwarp();
    tmem_alloc(&tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_launch_dependents();
  // (the builders wait inside their build; the producers, with `early`,
  // after their stages)
  const bool builder = warp >= kExpWarp0 && warp < kProducerWarp0;
  const bool epilogue = warp >= kEpiWarp0 && warp < kExpWarp0;
  // (with bstream the producers copy B rows the preceding grid writes: they
  // wait for it before their first stage)
  const bool early = p.early && !p.bstream;
  if (!builder && !epilogue && (warp < kProducerWarp0 || !early)) pdl_wait();
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp >= kProducerWarp0) {
    if (lane == 0) {
      // Producer x: stages i = x (mod 4), stage i = (unit u, j) being the
      // slabs (tile, 2 b) .. (tile, 2 b' - 1) of its blocks [b, b'), adjacent
      // in the tiled layout, into ring slot i mod ring (round r = i / ring).
      const int x = warp - kProducerWarp0;
      int last_i = -1, u = 0, j = x, slot = x, r = 0;
      while (j >= spu) { j -= spu; ++u; }
      const uint64_t pol = l2_policy_evict_first();   // codes are read once per call
      bool waited = !early;
      for (int i = x; i < nstages && ok; i += kExpSets) {
        // with `early`, kEarlyStages stages ahead of the preceding grid: more
        // would queue ahead of the loads that grid and this CTA's prologue
        // make once it completes
        if (!waited && i >= x + kExpSets * kEarlyStages) { pdl_wait(); waited = true; }
        if (r > 0) ok = mbar_wait(&c_empty[slot], (r - 1) & 1);
        if (!ok) break;
        const int b0 = sblk[j], b1 = sblk[j + 1];
        const int tile = prow + (u + rot < nunits ? u + rot : u + rot - nunits) * p.P;
        const uint8_t* src = reinterpret_cast<const uint8_t*>(p.codes) +
                             ((size_t)tile * p.KB + kb0 + b0) * p.blk_bytes;
        const uint32_t bytes = (uint32_t)(b1 - b0) * p.blk_bytes;
        uint8_t* dst = ring + (size_t)slot * p.slot_bytes;
        if (p.bstream) {
          // the stage's image pairs and scale words (L2 hits: the prepare
          // kernel wrote them, every CTA of the k chunk reads them)
          const int pa0 = (kb0 + b0) >> 1, pa1 = (kb0 + b1 + 1) >> 1;
          const uint32_t bb = (uint32_t)(pa1 - pa0) * (uint32_t)p.NP * 128u;
          const uint32_t sbytes = (uint32_t)(b1 - b0) * (uint32_t)p.NP * 4u;
          mbar_expect_tx(&c_full[slot], bytes + bb + sbytes);
          bulk_g2s_hint(dst, src, bytes, &c_full[slot], pol);
          bulk_g2s(dst + p.boff, p.bimg + (size_t)pa0 * p.NP * 128, bb, &c_full[slot]);
          bulk_g2s(dst + p.soff, p.sfbw + (size_t)(kb0 + b0) * p.NP * 4, sbytes, &c_full[slot]);
        } else {
          mbar_expect_tx(&c_full[slot], bytes);
          bulk_g2s_hint(dst, src, bytes, &c_full[slot], pol);
        }
        last_i = i;
        j += kExpSets;
        while (j >= spu) { j -= spu; ++u; }
        slot += kExpSets;
        if (slot >= p.ring) { slot -= p.ring; ++r; }
      }
      if (!waited) pdl_wait();
      // Every copy this thread issued has landed before the CTA may exit.
      for (int i = last_i; i >= 0 && i > last_i - p.ring; i -= kExpSets)
        if (!mbar_wait(&c_full[i % p.ring], (i / p.ring) & 1)) ok = false;
    }
  } else if (warp < kMaxPipes) {
    if (lane == 0 && warp < np) {
      // MMA issuer of pipeline e: stages i = e (mod np) in order, stage i's
      // codes in TMEM slot i mod 8, into the pipeline's accumulator.
      const int e = warp;
      ok = mbar_wait(&b_full, 0);
      tc_fence_after();
      const uint32_t idesc0 = mxf4_idesc(p.NP), idesc1 = idesc0 | (2u << 4);   // B scale bytes 0-1 / 2-3
      // Per stage: one wait, 2 nb MMAs, one commit; stage bookkeeping is
      // kept incremental (a single thread's scalar latency is on the path).
      const uint64_t bd0 = sw128_desc(sbase);
      const uint32_t ring_s = smem_u32(ring);
      const uint64_t astep = (uint64_t)((p.brow * 128) >> 4);   // descriptor units per image row pair
      const uint32_t sfa = tmem + (uint32_t)p.sfa, sfs = tmem + (uint32_t)p.sfs;
      const uint32_t sslot = (uint32_t)p.sss;   // B scale columns per TMEM slot
      const uint32_t aslot = (uint32_t)(kAColsPerBlk * p.sb);
      int k = 0, buf = 0, u = e / spu, j = e - (e / spu) * spu, last = -1;
      bool first = true;
      uint32_t dt = 0;
      for (int i = e; i < nstages && ok; i += np) {
        if (first) {
          buf = p.nbuf == 2 ? (k & 1) : 0;
          if (k >= p.nbuf) {
            ok = mbar_wait(&acc_empty[e][buf], ((k / p.nbuf) - 1) & 1);
            if (!ok) break;
          }
          dt = tmem + (uint32_t)(p.dbase + (e * p.nbuf + buf) * p.NP);
        }
        const int s = i & (p.ns - 1);
        ok = mbar_wait(&a_full[s], (i >> p.ns_log2) & 1);
        if (!ok) break;
        tc_fence_after();
        const int b0 = sblk[j], nb = sblk[j + 1] - b0;
        uint32_t at = tmem + (uint32_t)s * aslot;
        uint32_t sfb = sfs + (uint32_t)s * sslot;
        const int rslot = i % p.ring;
        // B rows: the chunk's resident image, or (bstream) the stage's pairs
        // in its ring slot
        const uint64_t bdb = p.bstream ? sw128_desc(ring_s + (uint32_t)rslot * p.slot_bytes + p.boff) : bd0;
        const int pbase = p.bstream ? (kb0 + b0) >> 1 : kb0 >> 1;
        for (int bb = 0; bb < nb; ++bb, at += kAColsPerBlk, sfb += (uint32_t)p.ss) {
          const int bl = b0 + bb, kb = kb0 + bl;
          const uint64_t bd = bdb + (uint64_t)((kb >> 1) - pbase) * astep + 4u * (uint32_t)(kb & 1);
          umma_mxf4_ts(dt, at, bd, idesc0, sfa, sfb, (first && bb == 0) ? 0u : 1u);
          umma_mxf4_ts(dt, at + 8, bd + 2, idesc1, sfa, sfb, 1u);
        }
        umma_commit(&a_empty[s]);
        if (p.bstream) umma_commit(&c_empty[rslot]);
        last = i;
        const int u0 = u;
        j += np;
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
      for (int i = last; i >= 0 && i > last - p.ns; i -= np)
        if (!mbar_wait(&a_empty[i & (p.ns - 1)], (i >> p.ns_log2) & 1)) ok = false;
    }
  } else if (warp >= kExpWarp0) {
    // ------------------------------------------------ builders, then expanders
    const int et = tid - 32 * kExpWarp0;
    pdl_wait();
    if (p.bstream) {
      // (the B rows and scale words arrive with each stage)
    } else if (p.bsrc == 2) {
      // The prepared image rows of the chunk's blocks and their scale words,
      // with 16-byte cp.async copies, all in flight at once (L2 hits: the
      // prepare kernel just wrote them).  A bulk copy here would queue behind
      // the code stream the producers have started on the same SM,
      // microseconds of HBM traffic.
      const int a0 = kb0 >> 1, a1 = (kb0 + ncb - 1) >> 1;
      if (p.brow == p.NP) {
        copy_lsu(reinterpret_cast<uint4*>(bop), reinterpret_cast<const uint4*>(p.bimg + (size_t)a0 * p.NP * 128),
                 (a1 - a0 + 1) * p.NP * 8, et);
      } else {   // the first 8 rows (1 KB) of every pair
        const uint4* src = reinterpret_cast<const uint4*>(p.bimg + (size_t)a0 * p.NP * 128);
        uint4* dst = reinterpret_cast<uint4*>(bop);
        for (int t = et; t < (a1 - a0 + 1) * 64; t += kBuildThreads)
          cp_async16(dst + t, src + (size_t)(t >> 6) * (p.NP * 8) + (t & 63), 16);
      }
      copy_lsu(reinterpret_cast<uint4*>(sfbs), reinterpret_cast<const uint4*>(p.sfbw + (size_t)kb0 * p.NP * 4),
               ncb * p.NP / 4, et);
      cp_async_wait_all();
    } else {
      write_terms(p, bop, sfbs, kb0, ncb, et);
    }
    fence_proxy_async_smem();   // generic-proxy stores -> the MMAs' async-proxy reads
    // A's scales, 1.0 for every row and K group: kSfaCols columns from sfa
    // (the B scales go with each stage, below)
    if (warp < kExpWarp0 + 4) {
      const uint32_t one[4] = {kUnitScales, kUnitScales, kUnitScales, kUnitScales};
      tmem_st4(tmem + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)p.sfa, one);
      tmem_st_wait();
    }
    tc_fence_before();
    named_bar_sync(3, kBuildThreads);
    if (et == 0) mbar_arrive(&b_full);   // (every issuer waits on its one phase)

    // Set x expands stages i = x (mod 4) in order: ring slot i mod ring,
    // TMEM slot i mod ns (its codes, then its B scales).
    const int x = (warp - kExpWarp0) >> 2, q = warp & 3, r = 32 * q + lane;
    const int MT = p.M * p.T;
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * q) << 16);
    const uint32_t aslot = (uint32_t)(kAColsPerBlk * p.sb);
    const uint32_t slab = p.blk_bytes / 2;
    int u = 0, j = x, slot = x, rnd = 0;
    while (j >= spu) { j -= spu; ++u; }
    for (int i = x; i < nstages && ok; i += kExpSets) {
      const int s = i & (p.ns - 1);
      ok = warp_wait(&c_full[slot], rnd & 1);
      if (!ok) break;
      // Codes into registers first, so that the ring slot goes back to the
      // producer before this set waits for its TMEM slot.
      const int sb0 = sblk[j], nb = sblk[j + 1] - sb0;
      j += kExpSets;
      while (j >= spu) { j -= spu; ++u; }
      const uint8_t* cs = ring + (size_t)slot * p.slot_bytes;
      uint32_t w[kMaxSb][8];
#pragma unroll
      for (int bb = 0; bb < kMaxSb; ++bb) {
        if (bb < nb) {
          const uint8_t* cb = cs + bb * p.blk_bytes;
          if constexpr (kTernary) {
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
      if (lane == 0 && !p.bstream) mbar_arrive(&c_empty[slot]);
      // (bstream: the slot's scale words are read below; the MMAs release it)
      const uint32_t* sws = p.bstream ? reinterpret_cast<const uint32_t*>(cs + p.soff)
                                      : reinterpret_cast<const uint32_t*>(sfbs) + (size_t)sb0 * p.NP;
      slot += kExpSets;
      if (slot >= p.ring) { slot -= p.ring; ++rnd; }
      if (i >= p.ns) {
        ok = warp_wait(&a_empty[s], ((i >> p.ns_log2) - 1) & 1);
        if (!ok) break;
        tc_fence_after();
      }
      // Few, wide TMEM stores: a tcgen05.st costs its warp a few hundred
      // cycles here whatever its width.  The codes first, two blocks per
      // store ...
#pragma unroll
      for (int bp = 0; bp < kMaxSb; bp += 2) {
        if (bp < nb) {
          // e2m1 nibble [sign, code bit 0, 0, 0]: +-2.0 or 0 (decode_stage_k order)
          uint32_t v[32];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int bb = bp + h;
            if constexpr (kTernary) {
#pragma unroll
              for (int wi = 0; wi < 8; ++wi) {
                v[16 * h + 2 * wi] = (w[bb][wi] << 2) & 0xCCCCCCCCu;   // even codes
                v[16 * h + 2 * wi + 1] = w[bb][wi] & 0xCCCCCCCCu;      // odd codes
              }
            } else {   // words hold the inverted bits: 1 = -1
#pragma unroll
              for (int wi = 0; wi < 4; ++wi)
#pragma unroll
                for (int k = 0; k < 4; ++k)
                  v[16 * h + 4 * wi + k] = ((w[bb][wi] << (3 - k)) & 0x88888888u) | 0x44444444u;
            }
          }
          const uint32_t ad = lane_addr + (uint32_t)s * aslot + (uint32_t)(kAColsPerBlk * bp);
          if (bp + 1 < nb) {
            tmem_st32(ad, v);
          } else {
            uint32_t v16[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v16[i] = v[i];
            tmem_st16(ad, v16);
          }
        }
      }
      // ... then the stage's B scales (one store for the slot when a block's
      // set is 4 columns)
      const uint32_t sc = lane_addr + (uint32_t)p.sfs + (uint32_t)(s * p.sss);
      if (p.ss == 4) {
        // column 4 bb + c: term row n = 32 c + lane of block bb; the slot's
        // scale area is sss = 4, 8 or 16 columns, one store of that width
        uint32_t sv[4 * kMaxSb];
#pragma unroll
        for (int cc = 0; cc < 4 * kMaxSb; ++cc) {
          const int bb = cc >> 2, n = 32 * (cc & 3) + lane;
          sv[cc] = (bb < nb && n < MT) ? sws[bb * p.NP + n] : kUnitScales;
        }
        if (p.sss == 16) {
          tmem_st16(sc, sv);
        } else if (p.sss == 8) {
          const uint32_t s8[8] = {sv[0], sv[1], sv[2], sv[3], sv[4], sv[5], sv[6], sv[7]};
          tmem_st8(sc, s8);
        } else {
          const uint32_t s4[4] = {sv[0], sv[1], sv[2], sv[3]};
          tmem_st4(sc, s4);
        }
      } else {
        for (int bb = 0; bb < nb; ++bb) {
          const uint32_t* sw = sws + (size_t)bb * p.NP;
          for (int c = 0; 32 * c < p.NP; ++c) {
            const int n = 32 * c + lane;
            tmem_st1(sc + (uint32_t)(bb * p.ss + c), n < MT ? sw[n] : kUnitScales);
          }
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[s]);
    }
  } else {
    // ------------------------------------------------------------- epilogue
    const int q = warp & 3, r = 32 * q + lane, et = tid - 32 * kEpiWarp0;
    const int NR = p.ntiles * kTileRows;
    const int MT = p.M * p.T;
    // alpha of this thread's row, fetched kAlphaAhead row tiles ahead into
    // a shared-memory ring by cp.async (one group per tile): a global load
    // issued while the code stream runs waits behind it for microseconds,
    // and a register it targets would stall the first instruction to touch
    // it.
    auto alpha_fetch = [&](int u) {
      if (u < nunits) {
        const int ut = u + rot < nunits ? u + rot : u + rot - nunits;
        const int row = (prow + ut * p.P) * kTileRows + r;
        if (row < p.n_out) cp_async4(&s_alpha[u % kAlphaAhead][et], p.alpha + row);
      }
      cp_async_commit();
    };
#pragma unroll
    for (int k = 0; k < kAlphaAhead; ++k) alpha_fetch(k);
    pdl_wait();   // y and the workspace belong to the preceding grid until then
    call_record_start(p.rec, p.call, blockIdx.x == 0 && et == 0);
    // the k-chunk-0 CTA of each row set puts this call's tag into the row
    // set's tickets while the main loop runs
    if (p.S > 1 && !p.atomic_y && sidx == 0 && et < 32)
      for (int u = et; u < nunits; u += 32) ticket_install(p.cnt + prow + u * p.P, p.call);
    int kc[kMaxPipes] = {0, 0, 0, 0};
    const uint32_t lq = tmem + ((uint32_t)(32 * q) << 16);
    for (int u = 0; u < nunits && ok; ++u) {
      // pipelines with stages in this tile: all, unless it has fewer stages
      uint32_t in = 0;
      if (spu >= np) {
        in = (1u << np) - 1u;
      } else {
        for (int t = 0; t < spu; ++t) in |= 1u << ((u * spu + t) % np);
      }
      bool w = true;
#pragma unroll
      for (int e = 0; e < kMaxPipes; ++e)
        if (((in >> e) & 1u) && w) w = mbar_wait(&acc_full[e][kc[e] % p.nbuf], (kc[e] / p.nbuf) & 1);
      ok = group_and(2, 128, w);
      if (!ok) break;
      tc_fence_after();
      const int ut = u + rot < nunits ? u + rot : u + rot - nunits;   // unit of this tile
      const int row = (prow + ut * p.P) * kTileRows + r;
      const bool live = row < p.n_out;
      cp_async_wait_group<kAlphaAhead - 1>();   // tile u's group has landed
      const float sa = live ? 0.5f * s_alpha[u % kAlphaAhead][et] : 0.f;
      alpha_fetch(u + kAlphaAhead);
      // y (or the partial) of batch row m from the sum of its T terms
      // where and how this tile's results are written (one address rule and
      // one kind of write per tile)
      const bool partial = p.S > 1 && !p.atomic_y;
      float* eb = partial ? p.part + (size_t)sidx * p.M * NR + row : p.y + row;
      uint32_t est = partial ? (uint32_t)NR : (uint32_t)p.n_out;
      float esc = partial ? 1.f : sa;
      int emode = !(partial || live) ? 0 : (p.atomic_y ? 1 : 2);   // none, float add, store
      int Mv = p.M;
      // (computed here, once: without this the compiler re-derives them from
      // the kernel parameters inside the loops below)
      asm volatile("" : "+l"(eb), "+r"(est), "+f"(esc), "+r"(emode), "+r"(Mv));
      auto emit = [&](int m, float acc) {
        if (m < Mv) {
          float* a = eb + (size_t)m * est;
          if (emode == 1) red_add_f32(a, esc * acc);
          else if (emode == 2) *a = esc * acc;
        }
      };
      // columns c0 .. c0 + 15 of the pipelines' accumulators, added (whole
      // x16 loads stay inside the NP columns, a multiple of 16); the
      // accumulators go back to the MMAs after the tile's last load
      auto load16 = [&](int c0, float (&sum)[16]) {
#pragma unroll
        for (int i = 0; i < 16; ++i) sum[i] = 0.f;
#pragma unroll
        for (int e = 0; e < kMaxPipes; ++e) {
          if ((in >> e) & 1u) {
            uint32_t rr[16];
            tmem_ld16(lq + (uint32_t)(p.dbase + (e * p.nbuf + kc[e] % p.nbuf) * p.NP + c0), rr);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) sum[i] += __uint_as_float(rr[i]);
          }
        }
        if (c0 + 16 >= MT) {
          tc_fence_before();
#pragma unroll
          for (int e = 0; e < kMaxPipes; ++e)
            if ((in >> e) & 1u) mbar_arrive(&acc_empty[e][kc[e] % p.nbuf]);
        }
      };
      if (MT <= 8) {
        // one batch row: 8 columns of two pipelines' accumulators in flight
        // per wait (the last tile's epilogue is the call's tail)
        float acc = 0.f;
#pragma unroll
        for (int e0 = 0; e0 < kMaxPipes; e0 += 2) {
          const bool h0 = (in >> e0) & 1u, h1 = (in >> (e0 + 1)) & 1u;
          uint32_t r0[8], r1[8];
          if (h0) tmem_ld8(lq + (uint32_t)(p.dbase + (e0 * p.nbuf + kc[e0] % p.nbuf) * p.NP), r0);
          if (h1) tmem_ld8(lq + (uint32_t)(p.dbase + ((e0 + 1) * p.nbuf + kc[e0 + 1] % p.nbuf) * p.NP), r1);
          if (h0 || h1) tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            if (h0 && i < MT) acc += __uint_as_float(r0[i]);
            if (h1 && i < MT) acc += __uint_as_float(r1[i]);
          }
        }
        tc_fence_before();
#pragma unroll
        for (int e = 0; e < kMaxPipes; ++e)
          if ((in >> e) & 1u) mbar_arrive(&acc_empty[e][kc[e] % p.nbuf]);
        emit(0, acc);
      } else if (MT <= 16) {
        // two batch rows: a short loop (not unrolled: it runs once per long
        // tile, and unrolled code is cold instruction memory every time, each
        // miss an L2 round trip while the code stream loads it)
        float sum[16];
        load16(0, sum);
        int m = 0, t = 0;
        float acc = 0.f;
#pragma unroll 1
        for (int i = 0; i < MT; ++i) {
          acc += sum[i];
          if (++t == p.T) { emit(m, acc); acc = 0.f; t = 0; ++m; }
        }
      } else {
        // many batch rows: 16 kSub columns hold whole rows, so where each
        // row's terms end is known at compile time and the sums stay in
        // registers (a loop over a register array indexed at run time puts
        // it in local memory: about 200 cycles a column)
        auto terms = [&](auto tc) {
          constexpr int T = decltype(tc)::value;
          constexpr int kSub = T == 4 ? 1 : 3;
          int m = 0;
          float acc = 0.f;
#pragma unroll 1
          for (int c0 = 0; c0 < MT; c0 += 16 * kSub) {
#pragma unroll
            for (int sub = 0; sub < kSub; ++sub) {
              const int cs = c0 + 16 * sub;
              if (cs < MT) {
                float sum[16];
                load16(cs, sum);
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                  acc += sum[i];
                  if ((16 * sub + i) % T == T - 1) {
                    emit(m, acc);
                    acc = 0.f;
                    ++m;
                  }
                }
              }
            }
          }
        };
        if (p.T == 3) terms(std::integral_constant<int, 3>());
        else if (p.T == 4) terms(std::integral_constant<int, 4>());
        else terms(std::integral_constant<int, 6>());
      }
#pragma unroll
      for (int e = 0; e < kMaxPipes; ++e) kc[e] += (in >> e) & 1u;
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
    __syncwarp();   // warp-collective: lane 0 ran the issuer loop alone
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

// Launch shape for batch M: the pipelines, TMEM slots, accumulators, stage
// size and (S, P) grid of at most one CTA per SM (more only where nothing
// else fits) that minimise a time model fitted to per-stage timestamps of
// the kernel: per CTA the stage rate of its MMA pipelines (about 150 cycles
// per MMA and 550 per stage on an issuing thread, the pipelines side by
// side) and of its 4 expander sets (a set waits for the MMAs of its
// previous stage when it owns one TMEM slot), against the HBM time of the
// codes (the bytes in flight capped by the CTAs' code rings, at a loaded
// latency), plus the prologue (B operand and scales) and the split-K tail.
// TMEM holds, from column 0: ns A slots of sb blocks (16 sb columns each),
// the A scales (4 columns), per slot the B scales of its sb blocks (a set of
// ss = 4 ceil(ceil(NP / 32) / 4) columns per block: scale columns start on a
// multiple of 4), and at the top the accumulators (npipe x nbuf x NP
// columns).
DecodeConfig decode_config_search(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  DecodeConfig best{};
  best.M = M;
  best.T = decode_terms(M);
  best.NP = (M * best.T + 15) / 16 * 16;
  best.ss = 4 * (((best.NP + 31) / 32 + 3) / 4);
  const int brow = decode_image(pl) && M * best.T <= 8 ? 8 : best.NP;
  const int KB = (int)(g.k_eff_pad / kBlk);
  const int sms = std::max(1, pl->sm_count);
  const int blk_bytes = kTileRows * kBlk * g.bits / 8;
  const double clk = 1.9e9;
  const double hbm = 6.0e12, cta_bw = 30e9;                    // bytes/s: HBM, one CTA's copy ring
  const double l2_bw = 20e12;                                  // bytes/s: L2 reads of streamed B rows
  const double t_tail = 2.0e-6, ring_latency = 4.0e-6;   // a ring slot's round trip under load
  const double c_mma = 150.0 + 0.5 * best.NP, c_stage = 550.0;   // issuing thread, cycles
  const double c_xblk = 200.0, c_xstage = 600.0;                 // expander set, cycles
  double best_t = 1e30;
  const int pipes[3] = {4, 2, 1};
  const int MT = M * best.T;
  double t_epi[3];
  for (int pi = 0; pi < 3; ++pi)
    t_epi[pi] = MT <= 16 ? 0.0   // (one or two batch rows: within the fitted per-tile cost below)
                         : ((MT + 15) / 16) * (385.0 * pipes[pi] + 650.0) / clk;
  // bstream 1: the stage's B rows and scale words stream into its ring slot
  // (whole block pairs per stage); only where the prepare kernel writes the
  // image, and for batches whose chunk-resident image would bound the k
  // chunk (M T > 8)
  for (int bs = 0; bs <= (decode_image(pl) && MT > 8 ? 1 : 0); ++bs)
  for (int pi = 0; pi < 3; ++pi) {
    const int np = pipes[pi];
    for (int ns = 4; ns <= kASlots; ns *= 2)
      for (int nbuf = 2; nbuf >= 1; --nbuf) {
        const int dbase = 512 - np * nbuf * best.NP;
        // k chunks beyond the SM count (CTAs in several waves) only where the
        // chunk's B operand and scales would not fit otherwise (large batches
        // on small parts)
        // TMEM slot: 16 sb code columns and its B scale columns (sb sets of
        // ss; with ss = 4 rounded up to 4, 8 or 16, the width of the one
        // store that writes them); then A's scales
        int sb = kMaxSb, sss = 0;
        for (; sb >= 1; --sb) {
          if (bs && (sb & 1)) continue;
          sss = best.ss == 4 ? (sb == 1 ? 4 : (sb == 2 ? 8 : 16)) : sb * best.ss;
          if (ns * (kAColsPerBlk * sb + sss) + kSfaCols <= dbase) break;
        }
        if (sb < 1) continue;                                    // TMEM
        for (int S = 1; S <= KB && (S <= sms || best.S == 0); ++S) {
          int CB = (KB + S - 1) / S;
          if (bs && S > 1) CB += CB & 1;                         // chunks start on a block pair
          if ((S - 1) * CB >= KB) continue;                      // no empty chunk
          const int b_bytes = bs ? 0 : (CB / 2 + 1) * brow * 128;    // image rows of the chunk's blocks
          const int sfb_bytes = bs ? 0 : (CB * best.NP * 4 + 15) / 16 * 16;  // its B scale words
          const int code_slot = sb * blk_bytes;
          const int bslot = (sb / 2) * best.NP * 128 + sb * best.NP * 4;    // streamed B rows + scales
          const int slot_bytes = bs ? (code_slot + bslot + 1023) / 1024 * 1024 : code_slot;
          // code bytes in flight per CTA: about the SM's share of HBM
          // bandwidth at the loaded latency, at least two stages per set
          int ring = std::min(kMaxRing, (kSmemMax - 2048 - b_bytes - sfb_bytes) / slot_bytes);
          ring = std::min(ring, std::max(2 * kExpSets, (kRingBytes + code_slot - 1) / code_slot + kExpSets - 1));
          ring -= ring % kExpSets;          // each ring slot belongs to one expander set
          if (ring < kExpSets) continue;
          const int npr = (CB + 1) / 2;
          const int spu = bs ? std::max((2 * npr + sb - 1) / sb, std::min(2, npr))
                             : std::max((CB + sb - 1) / sb, std::min(2, CB));
          if (spu > kMaxSpu) continue;
          const double issue = 2.0 * sb * c_mma + c_stage;        // cycles per stage, one pipeline
          const double expand = c_xstage + c_xblk * sb;           // cycles per stage, one set
          const double set_cyc = ns == 4 ? std::max(expand, issue * 4.0 / np + 300.0) : std::max(expand, issue * 2.0 / np);
          const double mma_rate = std::min(np / issue, kExpSets / set_cyc) * clk;   // stages per second per CTA
          // the prologue: the wait for the prepare kernel, the B operand (image
          // copy or terms formed in the CTA)
          const double t_build = bs ? 2.0e-6 : 2.0e-6 + (b_bytes + sfb_bytes) / 25e9 + CB * M * best.T * 2.0e-9;
          for (int P = 1; P <= std::min(g.ntiles, std::max(1, sms / S)); ++P) {
            const int grid = S * P;
            const int waves = (grid + sms - 1) / sms;
            const int units = (g.ntiles + P - 1) / P;
            // A CTA streams its units row tiles (CB blocks each) at the
            // lowest of: the measured per-CTA ceiling of the copy ring, its
            // share of HBM bandwidth, and the rate its MMA pipelines and
            // expander sets sustain (and, streaming B, its share of the L2's
            // bandwidth for the B rows); every row tile adds a cost that grows
            // with the k chunks adding into the same rows of y (accumulator
            // hand-off, epilogue, split-K contention: fitted to measured
            // calls), every call a prologue and a tail.
            const double tile_bytes = (double)CB * blk_bytes;
            double rate = std::min({cta_bw, hbm / std::min(grid, sms), mma_rate * code_slot,
                                    (double)ring * code_slot / ring_latency});
            if (bs) rate = std::min(rate, l2_bw / std::min(grid, sms) * code_slot / bslot);
            // the tile's epilogue (accumulator loads per pipeline and the
            // terms' sums and writes per 16 columns, measured per tile) runs
            // beside the next tile's MMAs with two accumulators, else between
            const double t_stream = tile_bytes / rate;
            const double t_tile = nbuf == 2 ? std::max(t_stream, t_epi[pi]) : t_stream + t_epi[pi];
            const double t_cta = units * (t_tile + 0.8e-6 + 0.15e-6 * S);
            const double t = waves * t_cta + t_build + t_tail;
            if (t < best_t * 0.999) {
              best_t = t;
              best.S = S; best.P = P; best.CB = CB; best.ring = ring; best.sb = sb;
              best.npipe = np; best.ns = ns; best.nbuf = nbuf; best.dbase = dbase; best.sss = sss;
              best.bstream = bs; best.brow = bs ? best.NP : brow;
              best.slot_bytes = slot_bytes; best.boff = code_slot; best.soff = code_slot + (sb / 2) * best.NP * 128;
              best.smem = std::max<size_t>(kSmemMin, 1024 + (size_t)b_bytes + sfb_bytes + (size_t)ring * slot_bytes);
            }
          }
        }
      }
  }
  best.sfa = best.ns * kAColsPerBlk * best.sb;
  best.sfs = best.sfa + kSfaCols;
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
  const int64_t v[16] = {dc.T, dc.NP, dc.S, dc.P, dc.CB, dc.ring, dc.sb, dc.nbuf, (int64_t)dc.smem,
                         dc.slot_bytes, dc.bstream ? 0 : (int64_t)(dc.CB / 2 + 1) * dc.brow * 128, dc.ss,
                         kSmemMax + 1024, dc.npipe, dc.ns, dc.bstream};
  for (int i = 0; i < 16; ++i) out[i] = v[i];
  return SDQ_OK;
}

namespace sdq {

bool decode_image(const sdq_plan_s* pl) { return pl->geo.n_b % 64 == 0; }


cudaError_t launch_decode(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st, int early, int y_mode) {
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
  p.sb = dc.sb; p.nbuf = dc.nbuf; p.npipe = dc.npipe; p.ns = dc.ns; p.ns_log2 = dc.ns == 8 ? 3 : 2;
  p.dbase = dc.dbase; p.sfa = dc.sfa; p.sfs = dc.sfs; p.ss = dc.ss; p.sss = dc.sss;
  p.n_out = g.n_out; p.ntiles = g.ntiles; p.ngroups = g.ngroups; p.ternary = g.bits == 2;
  p.early = early;
  p.atomic_y = y_mode == kYAdd || (y_mode == kYZeroed && dc.S > 1);
  p.blk_bytes = (uint32_t)(kTileRows * kBlk * g.bits / 8);
  p.slot_bytes = (uint32_t)dc.slot_bytes;
  p.bstream = dc.bstream; p.boff = (uint32_t)dc.boff; p.soff = (uint32_t)dc.soff;
  p.b_bytes = dc.bstream ? 0u : (uint32_t)((dc.CB / 2 + 1) * dc.brow * 128);
  p.brow = dc.brow;
  p.sfb_bytes = dc.bstream ? 0u : (uint32_t)((dc.CB * dc.NP * 4 + 15) / 16 * 16);
  static std::atomic<int> smem_set[64];   // per device: limit raised to kSmemMax + 1 KB
  static std::atomic<int> smem_set_b[64];
  cudaError_t e = p.ternary ? smem_limit_once(decode_kernel<true>, kSmemMax + 1024, pl->device, smem_set)
                            : smem_limit_once(decode_kernel<false>, kSmemMax + 1024, pl->device, smem_set_b);
  if (e != cudaSuccess) return e;
  return p.ternary ? launch_pdl(decode_kernel<true>, dim3(dc.S * dc.P), dim3(kThreads), dc.smem, st, p)
                   : launch_pdl(decode_kernel<false>, dim3(dc.S * dc.P), dim3(kThreads), dc.smem, st, p);
}

}  // namespace sdq
