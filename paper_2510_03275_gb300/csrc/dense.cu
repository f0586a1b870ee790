// K6 / K7: large-batch forward by rebuilding the layer's weights once per
// call, then one dense GEMM ("decimate, then dense").
//
//   W'[r, bB + k] = 2 sum_j c[r, b n_b + j] G[j, k]      (K6, per block b)
//   y[m, r]       = alpha_r / 2 sum_k W'[r, k] x[m, k]    (K7)
//
// equal to the code-domain forward y = alpha C x_tilde, x_tilde = G x per
// block (section 3.5, eq. 12), by associativity: C (G x) = (C G) x.  The
// code domain costs 2 M N K_eff flops; this route 2 M N K for the GEMM plus
// 4 N K_eff B for the rebuild (hi and lo parts of G), fewer when M exceeds
// about 2 OSR B / (OSR - 1).
//
// K6: the codes are the A operand in tensor memory (as in K5: exact bf16
// +-2 / 0 from one tcgen05.st per 64 codes), G^T the B operand, resident in
// shared memory for the CTA's lifetime (bf16 hi and lo parts, 128 output
// columns k x n_b codes, K-major, 128-byte swizzle, its K order permuted as
// the code expansion orders the codes); one 128 x 128 fp32 accumulator per
// (row tile, block) item, two of them so that an item's epilogue (bf16 W',
// 16-byte stores) overlaps the next item's MMAs.  Persistent CTAs over the
// items.
//   warp 0     TMEM allocation; lane 0: G^T once (TMA), then the code slabs
//   warp 1     lane 0: 8 MMAs per 64 codes (4 K steps x hi / lo)
//   warps 2-9  two expander sets (stages of one parity each)
//   warps 10-13 epilogue
// K7: a plain tcgen05 GEMM, D[r, m] = W' x^T per CTA tile of 128 (or 2 x 128)
// weight rows x 256 batch rows, both operands TMA-loaded (128-byte swizzle),
// 4 (3) stages; epilogue as K5's.
// Every wait on an mbarrier is bounded (about 2 s); a timeout writes the call
// number into the workspace's call record and the CTA finishes without
// further waits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBK = 64;                    // codes (K6) or inputs (K7) per stage

__device__ __forceinline__ void umma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate) : "memory");
}

// kind::f16 instruction descriptor: D fp32, A and B bf16, both K-major,
// M = 128, N = n.
__host__ __device__ constexpr uint32_t f16_idesc(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

// ---------------------------------------------------------------- K6 rebuild
constexpr int kRbStages = 6;
constexpr int kRbEpiWarp0 = 10;
constexpr int kRbThreads = 32 * 14;
constexpr int kRbCTile = 128 * 16;          // code slab of a stage: 128 rows x 64 codes, at most 2 KB
constexpr uint32_t kRbAcc = 128;            // accumulator columns (128 outputs k of a block)
constexpr uint32_t kRbAcol = 2 * kRbAcc;    // first A slot column
constexpr uint32_t kRbAslot = kBK / 2;

struct ReconParams {
  const uint32_t* codes;
  uint16_t* w;          // W', n_out x k_in bf16 row-major (rows past n_out not written)
  uint64_t* rec;
  uint64_t call;
  int n_out, k_in, nblk, n_b, ntiles, ngroups, wpg, quantizer, nitems;
};

__global__ void __launch_bounds__(kRbThreads, 1)
    recon_kernel(const __grid_constant__ CUtensorMap ghmap, const __grid_constant__ CUtensorMap glmap,
                 ReconParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t g_full, full[kRbStages], empty[kRbStages], a_full[kRbStages],
      acc_full[2], acc_empty[2];
  __shared__ uint32_t tmem_base;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  const int spb = p.n_b / kBK;                        // stages (64-code chunks) per block
  const uint32_t gchunk = 128u * 128u;                // one 64-code chunk of G^T: 128 rows x 128 B
  uint8_t* c_tiles = base + 2 * spb * gchunk;         // after G^T hi, lo
  const uint32_t slab_bytes = (uint32_t)(kTileRows * p.wpg * 4);

  if (tid == 0) {
    mbar_init(&g_full, 1);
    for (int s = 0; s < kRbStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&a_full[s], 4);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);
    }
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
  const uint32_t tmem = tmem_base;
  bool ok = true;
  // this CTA's items: (row tile, block) = item / nblk, item % nblk
  const int nmine = p.nitems > (int)blockIdx.x ? (p.nitems - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int nst = nmine * spb;

  if (warp == 0) {
    if (lane == 0) {
      mbar_expect_tx(&g_full, 2u * spb * gchunk);
      for (int c = 0; c < spb; ++c) {
        tma_load_2d(base + c * gchunk, &ghmap, c * kBK, 0, &g_full);
        tma_load_2d(base + (spb + c) * gchunk, &glmap, c * kBK, 0, &g_full);
      }
      for (int i = 0; i < nst && ok; ++i) {
        const int s = i % kRbStages, r = i / kRbStages;
        const int item = (int)blockIdx.x + (i / spb) * (int)gridDim.x, sc = i % spb;
        const int tile = item / p.nblk, b = item - tile * p.nblk;
        if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
        if (!ok) break;
        mbar_expect_tx(&full[s], slab_bytes);
        const uint32_t* src = p.codes + (size_t)((int64_t)tile * p.ngroups + b * spb + sc) * (slab_bytes / 4);
        bulk_g2s(c_tiles + s * kRbCTile, src, slab_bytes, &full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = f16_idesc(128);
      ok = mbar_wait(&g_full, 0);
      for (int i = 0; i < nst && ok; ++i) {
        const int s = i % kRbStages, r = i / kRbStages;
        const int it = i / spb, sc = i % spb, a = it & 1;
        if (sc == 0 && it >= 2) {
          ok = mbar_wait(&acc_empty[a], ((it >> 1) - 1) & 1);
          if (!ok) break;
        }
        ok = mbar_wait(&full[s], r & 1) && mbar_wait(&a_full[s], r & 1);
        if (!ok) break;
        tc_fence_after();
        const uint64_t bh = sw128_desc(sbase + sc * gchunk);
        const uint64_t bl = sw128_desc(sbase + (spb + sc) * gchunk);
        const uint32_t d = tmem + (uint32_t)a * kRbAcc;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
          const uint32_t at = tmem + kRbAcol + kRbAslot * s + 8 * kk;
          umma_f16_ts(d, at, bh + 2 * kk, idesc, (sc | kk) != 0);
          umma_f16_ts(d, at, bl + 2 * kk, idesc, 1u);
        }
        umma_commit(&empty[s]);
        if (sc == spb - 1) umma_commit(&acc_full[a]);
      }
    }
  } else if (warp < kRbEpiWarp0) {
    // Expanders: set x = (warp - 2) / 4 expands stages i = x (mod 2), thread
    // = code row 32 q + lane (q = warp % 4): 64 codes -> 32 TMEM columns.
    const int x = (warp - 2) >> 2, q = warp & 3, rr = 32 * q + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * q) << 16);
    for (int i = x; i < nst && ok; i += 2) {
      const int s = i % kRbStages, r = i / kRbStages;
      ok = mbar_wait(&full[s], r & 1);
      if (ok && r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);   // the slot's previous MMAs are done
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const uint8_t* cs = c_tiles + s * kRbCTile;
      uint32_t v[32];
      if (p.quantizer == SDQ_TERNARY) {
        const uint4 w4 = *reinterpret_cast<const uint4*>(cs + rr * 16);
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
          for (int j = 0; j < 8; ++j) v[8 * k + j] = (w[k] << (2 * j)) & 0xC000C000u;
      } else {   // words hold the inverted bits: 1 = -1
        const uint2 w2 = *reinterpret_cast<const uint2*>(cs + rr * 8);
        const uint32_t w[2] = {~w2.x, ~w2.y};
#pragma unroll
        for (int k = 0; k < 2; ++k)
#pragma unroll
          for (int j = 0; j < 16; ++j) v[16 * k + j] = ((w[k] << j) & 0x80008000u) | 0x40004000u;
      }
      tmem_st32(lane_addr + kRbAcol + kRbAslot * s, v);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[s]);
    }
  } else {
    // Epilogue: item it's accumulator -> W'[row, b B .. b B + 127] as bf16.
    const int q = warp & 3, rr = 32 * q + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * q) << 16);
    for (int it = 0; it < nmine && ok; ++it) {
      const int a = it & 1;
      ok = mbar_wait(&acc_full[a], (it >> 1) & 1);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const int item = (int)blockIdx.x + it * (int)gridDim.x;
      const int tile = item / p.nblk, b = item - tile * p.nblk;
      const int row = tile * kTileRows + rr;
      uint16_t* out = p.w + (size_t)row * p.k_in + (size_t)b * 128;
      for (int c0 = 0; c0 < 128; c0 += 32) {
        uint32_t u0[16], u1[16];
        tmem_ld16(lane_addr + (uint32_t)a * kRbAcc + (uint32_t)c0, u0);
        tmem_ld16(lane_addr + (uint32_t)a * kRbAcc + (uint32_t)c0 + 16, u1);
        tmem_ld_wait();
        if (c0 + 32 >= 128) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[a]);
        }
        if (row < p.n_out) {
          uint4* o = reinterpret_cast<uint4*>(out + c0);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t* u = h ? u1 : u0;
            o[2 * h] = make_uint4(pack_bf16x2(__uint_as_float(u[0]), __uint_as_float(u[1])),
                                  pack_bf16x2(__uint_as_float(u[2]), __uint_as_float(u[3])),
                                  pack_bf16x2(__uint_as_float(u[4]), __uint_as_float(u[5])),
                                  pack_bf16x2(__uint_as_float(u[6]), __uint_as_float(u[7])));
            o[2 * h + 1] = make_uint4(pack_bf16x2(__uint_as_float(u[8]), __uint_as_float(u[9])),
                                      pack_bf16x2(__uint_as_float(u[10]), __uint_as_float(u[11])),
                                      pack_bf16x2(__uint_as_float(u[12]), __uint_as_float(u[13])),
                                      pack_bf16x2(__uint_as_float(u[14]), __uint_as_float(u[15])));
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

// ------------------------------------------------------------ K7 dense GEMM
// WT = 1 or 2 weight tiles of 128 rows per CTA against one 256-row batch
// tile: with two, the x tile in shared memory serves two MMAs per K step
// (shared-memory traffic per MMA 136 instead of 163 bytes per cycle of tensor
// work), where the grid still fills the SMs.
constexpr int kDnBN = 256;
constexpr int kDnATile = 128 * kBK * 2;     // 16 KB: 128 weight rows x 64 inputs
constexpr int kDnBTile = kDnBN * kBK * 2;   // 32 KB: 256 batch rows x 64 inputs
constexpr int kDnThreads = 320;
template <int WT> struct DnShape {
  static constexpr int kStages = WT == 1 ? 4 : 3;
  static constexpr int kStage = WT * kDnATile + kDnBTile;
  static constexpr int kSmem = kStages * kStage + 1024;
  static constexpr uint32_t kCols = WT == 1 ? 256u : 512u;
};

struct DenseParams {
  const float* alpha;
  float* y;
  uint64_t* rec;
  uint64_t call;
  int M, N, nks;
  // CTA u < nfull takes unit u (weight-tile group u mod ngroups, batch tile u / ngroups, WT
  // tiles); CTAs from nfull on split the remaining units into their WT single tiles
  int ngroups, nfull;
};

template <int WT>
__global__ void __launch_bounds__(kDnThreads, 1)
    dense_kernel(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap xmap,
                 DenseParams p) {
  constexpr int kStages = DnShape<WT>::kStages, kStage = DnShape<WT>::kStage;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[kStages], empty[kStages], acc_bar;
  __shared__ uint32_t tmem_base;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int unit = blockIdx.x, nt = WT, sub = 0;
  if (unit >= p.nfull) {
    sub = (unit - p.nfull) % WT;
    unit = p.nfull + (unit - p.nfull) / WT;
    nt = 1;
  }
  const int n0 = (unit % p.ngroups) * 128 * WT + 128 * sub, m0 = (unit / p.ngroups) * kDnBN;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&acc_bar, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_base, DnShape<WT>::kCols);
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
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
        if (!ok) break;
        mbar_expect_tx(&full[s], (uint32_t)(nt * kDnATile + kDnBTile));
        uint8_t* st = base + s * kStage;
#pragma unroll
        for (int w = 0; w < WT; ++w)
          if (w < nt) tma_load_2d(st + w * kDnATile, &wmap, ks * kBK, n0 + 128 * w, &full[s]);
        tma_load_2d(st + WT * kDnATile, &xmap, ks * kBK, m0, &full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = f16_idesc(kDnBN);
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        ok = mbar_wait(&full[s], r & 1);
        if (!ok) break;
        tc_fence_after();
        const uint32_t st = sbase + s * kStage;
        const uint64_t bd = sw128_desc(st + WT * kDnATile);
#pragma unroll
        for (int w = 0; w < WT; ++w) {
          if (w >= nt) break;
          const uint64_t ad = sw128_desc(st + w * kDnATile);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            umma_bf16(tmem + (uint32_t)(w * kDnBN), ad + 2 * kk, bd + 2 * kk, idesc, (ks | kk) != 0);
        }
        umma_commit(&empty[s]);
      }
      umma_commit(&acc_bar);
    }
  } else {
    // Epilogue: lane quadrant q holds weight rows n0 + 128 w + 32 q + lane of
    // accumulator w; this warp writes its columns (batch rows) 128 h .. 128 h + 127.
    const int q = warp & 3, h = (warp - 2) >> 2, rr = 32 * q + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(32 * q) << 16);
    ok = mbar_wait(&acc_bar, 0);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
    if (ok) {
#pragma unroll 1
      for (int w = 0; w < nt; ++w) {
        const int row = n0 + 128 * w + rr;
        const float sa = row < p.N ? 0.5f * __ldg(p.alpha + row) : 0.f;
        for (int c0 = 128 * h; c0 < 128 * h + 128; c0 += 16) {
          uint32_t a[16];
          tmem_ld16(lane_addr + (uint32_t)(w * kDnBN + c0), a);
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
  }
  if (!ok) call_record_fail(p.rec, p.call);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, DnShape<WT>::kCols);
  }
}

}  // namespace

bool dense_route_applies(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  return M >= kDenseMinM && pl->d_gt_hi && g.block == 128 && g.n_b % kBK == 0 && g.n_b <= kDenseMaxNb &&
         g.k_in % 64 == 0;
}

cudaError_t launch_dense_forward(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha,
                                 const uint16_t* x, int M, float* y, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) || (g.k_in * 2) % 16) return cudaErrorNotSupported;
  auto enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
  if (!enc) return cudaErrorNotSupported;
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* wbase = static_cast<uint8_t*>(ws);
  uint16_t* wp = reinterpret_cast<uint16_t*>(wbase + L.what);
  const cuuint32_t estr[2] = {1, 1};
  const int spb = g.n_b / kBK;
  // K6: G^T hi / lo maps (128 rows x n_b), one 64-code chunk per box
  CUtensorMap ghmap, glmap, wmap, xmap;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)g.n_b, 128};
    const cuuint64_t strides[1] = {(cuuint64_t)g.n_b * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, 128};
    if (enc(&ghmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pl->d_gt_hi, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
        enc(&glmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, pl->d_gt_lo, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  // K7: W' (n_out x k_in, rows past n_out read as zeros) and x (M x k_in)
  {
    const cuuint64_t dims[2] = {(cuuint64_t)g.k_in, (cuuint64_t)g.n_out};
    const cuuint64_t strides[1] = {(cuuint64_t)g.k_in * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, 128};
    if (enc(&wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, wp, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)g.k_in, (cuuint64_t)M};
    const cuuint64_t strides[1] = {(cuuint64_t)g.k_in * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kDnBN};
    if (enc(&xmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(x), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  ReconParams rp;
  rp.codes = codes; rp.w = wp;
  rp.rec = reinterpret_cast<uint64_t*>(wbase + L.err);
  rp.call = call_tag(next_call_number());
  rp.n_out = g.n_out; rp.k_in = g.k_in; rp.nblk = g.nblk; rp.n_b = g.n_b; rp.ntiles = g.ntiles;
  rp.ngroups = g.ngroups; rp.wpg = g.wpg; rp.quantizer = pl->desc.quantizer;
  rp.nitems = g.ntiles * g.nblk;
  const size_t rsmem = 1024 + 2 * (size_t)spb * 128 * 128 + kRbStages * (size_t)kRbCTile;
  if (rsmem > 227 * 1024) return cudaErrorNotSupported;
  cudaError_t e = cudaFuncSetAttribute(recon_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rsmem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(recon_kernel, dim3(std::min(rp.nitems, std::max(1, pl->sm_count))), dim3(kRbThreads), rsmem, st,
                 ghmap, glmap, rp);
  if (e != cudaSuccess) return e;
  DenseParams dp;
  dp.alpha = alpha; dp.y = y;
  dp.rec = rp.rec;
  dp.call = call_tag(next_call_number());
  dp.M = M; dp.N = g.n_out; dp.nks = g.k_in / kBK;
  // two weight tiles per CTA where that still gives two waves of CTAs
  const int sms = std::max(1, pl->sm_count);
  const int mt = (M + kDnBN - 1) / kDnBN;
  if ((int64_t)((g.ntiles + 1) / 2) * mt >= 2 * sms) {
    dp.ngroups = (g.ntiles + 1) / 2;
    const int units = dp.ngroups * mt, waves = units / sms, rest = units - waves * sms;
    // a last wave of at most half the SMs runs as single tiles on twice the CTAs: the
    // wave then takes a single tile's time (~0.6 of a pair's) instead of a pair's
    dp.nfull = (rest > 0 && 2 * rest <= sms) ? waves * sms : units;
    const int grid = dp.nfull + 2 * (units - dp.nfull);
    e = cudaFuncSetAttribute(dense_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, DnShape<2>::kSmem);
    if (e != cudaSuccess) return e;
    return launch_pdl(dense_kernel<2>, dim3(grid), dim3(kDnThreads), (size_t)DnShape<2>::kSmem, st, wmap, xmap, dp);
  }
  dp.ngroups = g.ntiles;
  dp.nfull = g.ntiles * mt;
  e = cudaFuncSetAttribute(dense_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, DnShape<1>::kSmem);
  if (e != cudaSuccess) return e;
  return launch_pdl(dense_kernel<1>, dim3(dp.nfull), dim3(kDnThreads), (size_t)DnShape<1>::kSmem, st, wmap, xmap,
                    dp);
}

}  // namespace sdq
