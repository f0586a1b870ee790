// K5: prefill contraction (M > 64) on the 5th-generation tensor cores.
//
//   y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]        (section 3.5, eq. 12)
//
// A dense contraction over K_eff = OSR * K, run transposed as a bf16 GEMM
// with fp32 accumulation, D[r, m] = sum_j c[r, j] x_tilde[m, j]: the codes
// are the A operand in tensor memory, expanded from the packed 2-bit / 1-bit
// words to exact bf16 +-2.0 / 0 straight from registers by tcgen05.st (they
// never occupy shared memory: expanded into a shared-memory tile, their
// writes and the MMA's reads of them held the tensor pipe to ~60 %), and
// x_tilde (M x K_eff bf16, written by the prepare kernel in the permuted
// 64-code stage order the expansion yields) is the B operand, loaded by TMA
// in the canonical K-major 128-byte-swizzled layout.
//
// CTA tile 128 code rows (M of the MMA = TMEM lanes) x 256 batch rows (N),
// 64 codes per pipeline stage, kStages stages:
//   warp 0      TMEM allocation; lane 0 issues the TMA load of the stage's
//               x_tilde tile and the bulk copy of its code slab (tiled
//               layout: 128 rows x 64 codes, contiguous)
//   warp 1      lane 0 issues tcgen05.mma (4 x K = 16 per stage, A from the
//               stage's TMEM slot), commits to the stage's "empty" barrier,
//               finally to the accumulator one
//   warps 2..9  two expander sets (set x expands the stages of parity x),
//               thread = code row: its 64 codes become 32 TMEM columns of
//               bf16 pairs (one x32 store); then the epilogue: accumulator
//               column m -> y[m, r] scaled by alpha_r / 2, each warp one lane
//               quadrant and half of the 256 columns
// TMEM: accumulator columns 0..255, A slot s at 256 + 32 s.
// Every wait on an mbarrier is bounded (about 2 s); a timeout writes the call
// number into the workspace's call record and the CTA finishes without
// further waits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 6;
constexpr int kXTile = kBN * kBK * 2;     // 32 KB: 256 batch rows x 64 codes of bf16 x_tilde
constexpr int kCTile = kBM * 16;          // packed codes of a stage: 128 rows x 64 codes, at most 2 KB
constexpr int kSmem = kStages * (kXTile + kCTile) + 1024;
constexpr int kThreads = 320;   // 2 control warps + 8 expander / epilogue warps
constexpr uint32_t kAcol = kBN;           // first TMEM column of the A slots
constexpr uint32_t kAslot = kBK / 2;      // TMEM columns per A slot (bf16 pairs)

struct PrefillParams {
  const uint32_t* codes;
  const float* alpha;
  float* y;
  uint64_t* rec;       // call record
  uint64_t call;
  int M, N, ntiles, ngroups, wpg, nks, quantizer;
};

// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major,
// M = 128, N = 256.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                            ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ void umma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                             uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate) : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap xmap, PrefillParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[kStages], empty[kStages], a_full[kStages], acc_bar;
  __shared__ uint32_t tmem_base;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x, n0 = tile * kBM, m0 = blockIdx.y * kBN;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* x_tiles = base;
  uint8_t* c_tiles = base + kStages * kXTile;
  const uint32_t slab_bytes = (uint32_t)(kTileRows * p.wpg * 4);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&a_full[s], 4);
    }
    mbar_init(&acc_bar, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  pdl_launch_dependents();
  call_record_start(p.rec, p.call, blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0);
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp == 0) {
    if (lane == 0) {
      // Producer: TMA of the x_tilde tile [m0, m0 + 256) x [64 ks, 64 ks + 64)
      // (rows past M read as zeros) and the bulk copy of code slab (tile, ks).
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
        if (!ok) break;
        mbar_expect_tx(&full[s], kXTile + slab_bytes);
        tma_load_2d(x_tiles + s * kXTile, &xmap, ks * kBK, m0, &full[s]);
        const uint32_t* src = p.codes + (size_t)((int64_t)tile * p.ngroups + ks) * (slab_bytes / 4);
        bulk_g2s(c_tiles + s * kCTile, src, slab_bytes, &full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        ok = mbar_wait(&full[s], r & 1) && mbar_wait(&a_full[s], r & 1);
        if (!ok) break;
        tc_fence_after();
        const uint64_t bd = sw128_desc(sbase + s * kXTile);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
          umma_bf16_ts(tmem, tmem + kAcol + kAslot * s + 8 * kk, bd + 2 * kk, kIdesc, (ks | kk) != 0);
        umma_commit(&empty[s]);
      }
      umma_commit(&acc_bar);
    }
  } else {
    // Expanders: set x = (warp - 2) / 4 expands stages ks = x (mod 2); the
    // thread of lane quadrant q = warp % 4 expands code row 32 q + lane.
    const int x = (warp - 2) >> 2, q = warp & 3, rr = 32 * q + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * q) << 16);
    for (int ks = x; ks < p.nks && ok; ks += 2) {
      const int s = ks % kStages, r = ks / kStages;
      ok = mbar_wait(&full[s], r & 1);                         // the code slab has landed
      if (ok && r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);   // TMEM slot s: its MMAs are done
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const uint8_t* cs = c_tiles + s * kCTile;
      uint32_t v[32];
      if (p.quantizer == SDQ_TERNARY) {
        // 16 codes per word, code 2 bits: (w << 2 j) & 0xC000C000 puts two
        // codes into the sign and exponent-MSB bits of a bf16 pair (+-2 / 0)
        const uint4 w4 = *reinterpret_cast<const uint4*>(cs + rr * 16);
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 8; ++j) v[8 * i + j] = (w[i] << (2 * j)) & 0xC000C000u;
      } else {   // words hold the inverted bits: 1 = -1
        const uint2 w2 = *reinterpret_cast<const uint2*>(cs + rr * 8);
        const uint32_t w[2] = {~w2.x, ~w2.y};
#pragma unroll
        for (int i = 0; i < 2; ++i)
#pragma unroll
          for (int j = 0; j < 16; ++j) v[16 * i + j] = ((w[i] << j) & 0x80008000u) | 0x40004000u;
      }
      tmem_st32(lane_addr + kAcol + kAslot * s, v);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[s]);
    }
    // Epilogue: TMEM lane quadrant q holds code rows n0 + 32 q + lane; this
    // warp writes accumulator columns (batch rows) 128 x .. 128 x + 127.
    if (ok) ok = mbar_wait(&acc_bar, 0);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
    if (ok) {
      const int row = n0 + rr;
      const float sa = row < p.N ? 0.5f * __ldg(p.alpha + row) : 0.f;
      for (int c0 = 128 * x; c0 < 128 * x + 128; c0 += 16) {
        uint32_t a[16];
        tmem_ld16(lane_addr + (uint32_t)c0, a);
        tmem_ld_wait();
        if (row < p.N) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int m = m0 + c0 + i;
            if (m < p.M) p.y[(size_t)m * p.N + row] = __uint_as_float(a[i]) * sa;
          }
        }
      }
    }
  }
  if (!ok) call_record_fail(p.rec, p.call);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();   // warp-collective: lane 0 ran the producer loop alone
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// ------------------------------------------ prefill prepare, tensor cores
// x_tilde = G x_b for every block b (section 3.5), as one GEMM: x viewed as
// R = M nblk rows of B = 128 inputs (row r = block r mod nblk of batch row
// r / nblk), x_tilde rows = x rows . G^T (128 x n_b), on tcgen05.mma
// kind::f16 (M = 128 rows, N = n_b, K = 16 per instruction) with G split
// into bf16 hi and lo parts accumulated into the same fp32 accumulator (the
// pair carries G to ~2^-16; x is bf16, exact).  Persistent CTAs, one per SM,
// over tiles of 128 rows:
//   warp 0     TMEM allocation (two accumulators of n_b columns); lane 0
//              loads G hi / lo once, then the x tiles into a 3-slot ring
//              (TMA, 128-byte swizzle: the canonical K-major operand layout)
//   warp 1     lane 0 issues each tile's 16 MMAs into accumulator t mod 2
//   warps 2-9  epilogue, two warps per TMEM lane quadrant (half of the n_b
//              columns each): bf16 x_tilde (round to nearest even) in the
//              prefill operand order (prefill_pos64) with 16-byte stores;
//              the K padding of every batch row set to zero
// Layers with n_b above 256 take one launch per 256 or fewer columns (x read
// once per launch).  Bounded waits as in the contraction kernels.
constexpr int kPtEpiWarps = 8;
constexpr int kPtThreads = 64 + 32 * kPtEpiWarps;
constexpr int kPtRows = 128;
constexpr int kPtXTile = kPtRows * 128 * 2;   // 32 KB: 128 rows x 128 bf16 (two 64-wide K chunks)
constexpr int kPtSlots = 3;                   // x ring (with G hi / lo of n_b = 256: 225 KB)

struct PrepTcParams {
  uint16_t* xtb;
  uint64_t* rec;
  uint64_t call;
  int64_t R, k_eff, kpad;
  int M, nblk, n_b, ntile, ternary;
  int j0, ncol;   // this launch's x_tilde columns j0 .. j0 + ncol - 1 of every block (ncol <= 256)
};

__global__ void __launch_bounds__(kPtThreads, 1)
    prep_tc_kernel(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap ghmap,
                   const __grid_constant__ CUtensorMap glmap, PrepTcParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t g_full, x_full[kPtSlots], x_empty[kPtSlots], acc_full[2], acc_empty[2];
  __shared__ uint32_t tmem_base;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  const uint32_t gchunk = (uint32_t)p.ncol * 128u;  // one 64-wide K chunk of G^T: ncol rows x 128 B
  uint8_t* gh = base;                               // 2 chunks
  uint8_t* gl = base + 2 * gchunk;                  // 2 chunks
  uint8_t* xs = base + 4 * gchunk;                  // kPtSlots ring slots
  const uint32_t tcols = p.ncol <= 64 ? 128u : (p.ncol <= 128 ? 256u : 512u);

  if (tid == 0) {
    mbar_init(&g_full, 1);
    for (int s = 0; s < kPtSlots; ++s) {
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&acc_full[s], 1);
      mbar_init(&acc_empty[s], kPtEpiWarps);
    }
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_base, tcols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp == 0) {
    if (lane == 0) {
      // G (the plan's table, never written by the stream) before the wait
      // for the preceding grid; x and the workspace after it
      mbar_expect_tx(&g_full, 4 * gchunk);
      for (int c = 0; c < 2; ++c) {
        tma_load_2d(gh + c * gchunk, &ghmap, 64 * c, 0, &g_full);
        tma_load_2d(gl + c * gchunk, &glmap, 64 * c, 0, &g_full);
      }
      pdl_wait();
      pdl_launch_dependents();
      int i = 0;
      for (int t = blockIdx.x; t < p.ntile && ok; t += gridDim.x, ++i) {
        const int s = i % kPtSlots, r = i / kPtSlots;
        if (r > 0) ok = mbar_wait(&x_empty[s], (r - 1) & 1);
        if (!ok) break;
        mbar_expect_tx(&x_full[s], kPtXTile);
        tma_load_2d(xs + s * kPtXTile, &xmap, 0, t * kPtRows, &x_full[s]);
        tma_load_2d(xs + s * kPtXTile + kPtXTile / 2, &xmap, 64, t * kPtRows, &x_full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(p.ncol >> 3) << 17) |
                             ((uint32_t)(kPtRows >> 4) << 24);
      ok = mbar_wait(&g_full, 0);
      int i = 0;
      for (int t = blockIdx.x; t < p.ntile && ok; t += gridDim.x, ++i) {
        const int s = i % kPtSlots, r = i / kPtSlots, a = i & 1, ra = i >> 1;
        ok = mbar_wait(&x_full[s], r & 1);
        if (ok && ra > 0) ok = mbar_wait(&acc_empty[a], (ra - 1) & 1);
        if (!ok) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(a * p.ncol);
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint64_t ad = sw128_desc(sbase + 4 * gchunk + s * kPtXTile + c * (kPtXTile / 2));
          const uint64_t bh = sw128_desc(sbase + c * gchunk);
          const uint64_t bl = sw128_desc(sbase + (2 + c) * gchunk);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            umma_bf16(d, ad + 2 * kk, bh + 2 * kk, idesc, (c | kk) != 0);
            umma_bf16(d, ad + 2 * kk, bl + 2 * kk, idesc, 1);
          }
        }
        umma_commit(&x_empty[s]);
        umma_commit(&acc_full[a]);
      }
    }
  } else {
    pdl_wait();   // the workspace belongs to the preceding grid until then
    const int et = tid - 64, q = warp & 3, half = (warp - 2) >> 2;
    // the K padding of every batch row (k_eff .. kpad, a multiple of 8; by
    // the launch of the first columns)
    if (p.j0 == 0)
    for (int64_t z = (int64_t)blockIdx.x * (32 * kPtEpiWarps) + et; z < (int64_t)p.M * ((p.kpad - p.k_eff) / 8);
         z += (int64_t)gridDim.x * (32 * kPtEpiWarps)) {
      const int64_t per = (p.kpad - p.k_eff) / 8, m = z / per;
      *reinterpret_cast<uint4*>(p.xtb + m * p.kpad + p.k_eff + 8 * (z - m * per)) = make_uint4(0, 0, 0, 0);
    }
    const int cw = p.ncol / 2;                                  // this warp's columns
    const uint32_t lq = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(half * cw);
    int i = 0;
    for (int t = blockIdx.x; t < p.ntile && ok; t += gridDim.x, ++i) {
      const int s = i & 1, r = i >> 1;
      ok = mbar_wait(&acc_full[s], r & 1);
      if (!ok) break;
      tc_fence_after();
      const int64_t row = (int64_t)t * kPtRows + 32 * q + lane;
      const bool live = row < p.R;
      const int64_t m = live ? row / p.nblk : 0;
      uint16_t* out = p.xtb + m * p.kpad + (live ? (row - m * p.nblk) * p.n_b : 0) + p.j0 + half * cw;
      const uint32_t acol = (uint32_t)(s * p.ncol);
      // 32 columns at a time: a ternary operand permutes within 16, a binary
      // one within 32 positions (prefill_pos64); physical pair (2k, 2k + 1)
      // of a 16 (32) holds logical 7 - k and 15 - k (15 - k and 31 - k)
      for (int c0 = 0; c0 < cw; c0 += 32) {
        uint32_t a[16], b[16];
        tmem_ld16(lq + acol + (uint32_t)c0, a);
        tmem_ld16(lq + acol + (uint32_t)c0 + 16, b);
        tmem_ld_wait();
        if (c0 + 32 >= cw) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[s]);
        }
        uint32_t w[16];
        if (p.ternary) {
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            w[k] = pack_bf16x2(__uint_as_float(a[7 - k]), __uint_as_float(a[15 - k]));
            w[8 + k] = pack_bf16x2(__uint_as_float(b[7 - k]), __uint_as_float(b[15 - k]));
          }
        } else {
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const float lo = k < 16 ? __uint_as_float(a[15 - k]) : 0.f;
            const float hi = __uint_as_float(b[15 - k]);
            w[k] = pack_bf16x2(lo, hi);
          }
        }
        if (live) {
          uint4* o = reinterpret_cast<uint4*>(out + c0);
          o[0] = make_uint4(w[0], w[1], w[2], w[3]);
          o[1] = make_uint4(w[4], w[5], w[6], w[7]);
          o[2] = make_uint4(w[8], w[9], w[10], w[11]);
          o[3] = make_uint4(w[12], w[13], w[14], w[15]);
        }
      }
    }
  }
  if (!ok) call_record_fail(p.rec, p.call);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();   // warp-collective: lane 0 ran the producer loop alone
    tc_fence_after();
    tmem_dealloc(tmem, tcols);
  }
}

}  // namespace

void* tensor_map_encoder() { return reinterpret_cast<void*>(encode_fn()); }

cudaError_t launch_prefill(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                           float* y, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* wbase = static_cast<uint8_t*>(ws);
  auto enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap amap;
  const cuuint64_t dims[2] = {(cuuint64_t)g.k_eff_pad, (cuuint64_t)M};
  const cuuint64_t strides[1] = {(cuuint64_t)g.k_eff_pad * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kBN};
  const cuuint32_t estr[2] = {1, 1};
  CUresult cr = enc(&amap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, wbase + L.xt, dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;
  PrefillParams p;
  p.codes = codes; p.alpha = alpha; p.y = y;
  p.rec = reinterpret_cast<uint64_t*>(wbase + L.err);
  p.call = call_tag(next_call_number());
  p.M = M; p.N = g.n_out; p.ntiles = g.ntiles; p.ngroups = g.ngroups; p.wpg = g.wpg;
  p.nks = (int)(g.k_eff_pad / kBK);
  p.quantizer = pl->desc.quantizer;
  cudaError_t e = cudaFuncSetAttribute(prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  dim3 grid(g.ntiles, (M + kBN - 1) / kBN);
  return launch_pdl(prefill_kernel, grid, dim3(kThreads), (size_t)kSmem, st, amap, p);
}


// The prefill prepare kernel on the tensor cores where it applies (B = 128,
// n_b a multiple of 64, x 16-byte aligned), one launch per 256 or fewer of
// the n_b columns; *used = false otherwise.
cudaError_t launch_prep_tc(const sdq_plan_s* pl, const uint16_t* x, int M, void* ws, cudaStream_t st,
                           bool* used) {
  const Geometry& g = pl->geo;
  *used = false;
  if (g.block != 128 || g.n_b % 64 != 0 || (reinterpret_cast<uintptr_t>(x) & 15u)) return cudaSuccess;
  auto enc = encode_fn();
  if (!enc) return cudaSuccess;
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* wbase = static_cast<uint8_t*>(ws);
  const int64_t R = (int64_t)M * g.nblk;
  if (R >= (int64_t(1) << 31) - kPtRows) return cudaSuccess;
  const int nparts = (g.n_b + 255) / 256;
  CUtensorMap xmap, ghmap[16], glmap[16];
  if (nparts > 16) return cudaSuccess;
  const cuuint32_t estr[2] = {1, 1};
  {
    const cuuint64_t dims[2] = {128, (cuuint64_t)R};
    const cuuint64_t strides[1] = {256};
    const cuuint32_t box[2] = {64, (cuuint32_t)kPtRows};
    if (enc(&xmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(x), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaSuccess;
  }
  int j0s[16], ncols[16];
  for (int q = 0, j0 = 0; q < nparts; ++q) {
    const int ncol = std::min(256, g.n_b - j0);
    const cuuint64_t dims[2] = {128, (cuuint64_t)ncol};
    const cuuint64_t strides[1] = {256};
    const cuuint32_t box[2] = {64, (cuuint32_t)ncol};
    if (enc(&ghmap[q], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pl->d_g_hi + (size_t)j0 * 128, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
        enc(&glmap[q], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pl->d_g_lo + (size_t)j0 * 128, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaSuccess;
    j0s[q] = j0;
    ncols[q] = ncol;
    j0 += ncol;
  }
  PrepTcParams p;   // (a timeout is recorded under this kernel's own call number)
  p.xtb = reinterpret_cast<uint16_t*>(wbase + L.xt);
  p.rec = reinterpret_cast<uint64_t*>(wbase + L.err);
  p.R = R; p.k_eff = g.k_eff; p.kpad = g.k_eff_pad;
  p.M = M; p.nblk = g.nblk; p.n_b = g.n_b; p.ternary = pl->desc.quantizer == SDQ_TERNARY;
  p.ntile = (int)((R + kPtRows - 1) / kPtRows);
  const size_t smem_max = 1024 + 4 * (size_t)256 * 128 + kPtSlots * (size_t)kPtXTile;
  cudaError_t e = cudaFuncSetAttribute(prep_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_max);
  if (e != cudaSuccess) return e;
  const int grid = std::min(p.ntile, std::max(1, pl->sm_count));
  *used = true;
  for (int q = 0; q < nparts; ++q) {
    p.call = call_tag(next_call_number());
    p.j0 = j0s[q];
    p.ncol = ncols[q];
    const size_t smem = 1024 + 4 * (size_t)p.ncol * 128 + kPtSlots * (size_t)kPtXTile;
    e = launch_pdl(prep_tc_kernel, dim3(grid), dim3(kPtThreads), smem, st, xmap, ghmap[q], glmap[q], p);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}
}  // namespace sdq
