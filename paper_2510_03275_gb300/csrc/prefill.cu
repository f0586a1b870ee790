// K5: prefill contraction (M > 64) on the 5th-generation tensor cores.
//
//   y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]        (section 3.5, eq. 12)
//
// A dense contraction over K_eff = OSR * K, run as a bf16 GEMM with fp32
// accumulation: A = x_tilde (M x K_eff bf16, written by the prep kernel in
// the permuted 64-code stage order below), B = the codes (N x K_eff),
// expanded tile by tile from the packed 2-bit / 1-bit words to exact bf16
// values +-2.0 / 0 directly in shared memory, in the canonical K-major
// 128-byte-swizzled operand layout of tcgen05.mma.
//
// CTA tile 128 (M) x 256 (N), 64 codes per pipeline stage, kStages stages:
//   warp 0      TMEM allocation; lane 0 issues the TMA loads of the A tile
//               and of the packed code words of every stage
//   warp 1      lane 0 issues tcgen05.mma (4 x K=16 per stage), commits to
//               the stage's "empty" barrier, finally to the accumulator one
//   warps 2..9  expand the B tile of every stage (one 16-byte smem chunk per
//               8 codes of one row; the shift-and-mask expansion of a tiled
//               word yields its codes in the permuted order the prep kernel
//               also uses for A), then read the fp32 accumulator out of TMEM
//               (tcgen05.ld), scale by alpha / 2 and store y.
// Every wait on an mbarrier is bounded (about 2 s); a timeout sets the
// workspace error word and the CTA finishes without further waits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kATile = kBM * kBK * 2;     // 16 KB
constexpr int kBTile = kBN * kBK * 2;     // 32 KB
constexpr int kCTile = 16 * 64 * 4;       // packed codes of a stage: 16 row groups x 256 bytes
constexpr int kSmem = kStages * (kATile + kBTile + kCTile) + 1024;
constexpr int kThreads = 320;   // 2 control warps + 8 expander / epilogue warps
constexpr int kExp = 256;       // expander threads

struct PrefillParams {
  const uint32_t* codes;
  const float* alpha;
  float* y;
  uint32_t* err;
  int M, N, ng, n_chunks, nks, quantizer;
};

// ----------------------------------------------------------- PTX wrappers
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(dst)),
               "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate) : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                   smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar)) : "memory");
}
// 32 TMEM lanes x 16 columns of 32-bit values: register i of the thread of
// lane l holds (lane base + l, column + i).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
      " [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (SBO), start address in 16-byte units.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                 // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;       // stride byte offset
  d |= (uint64_t)1 << 46;                 // descriptor version
  d |= (uint64_t)2 << 61;                 // SWIZZLE_128B
  return d;
}

// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                            ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ void st_chunk(uint8_t* btile, int n, int c8, uint32_t a, uint32_t b,
                                         uint32_t c, uint32_t d) {
  uint4* p = reinterpret_cast<uint4*>(btile + n * 128 + ((c8 ^ (n & 7)) << 4));
  *p = make_uint4(a, b, c, d);
}

__global__ void __launch_bounds__(kThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap cmap,
                   PrefillParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_a[kStages], full_b[kStages], empty[kStages], acc_bar;
  __shared__ uint32_t tmem_base;
  __shared__ int fail;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * kBN, m0 = blockIdx.y * kBM;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* a_tiles = base;
  uint8_t* b_tiles = base + kStages * kATile;
  const uint32_t* c_tiles = reinterpret_cast<const uint32_t*>(base + kStages * (kATile + kBTile));
  const int cwords = p.quantizer == SDQ_TERNARY ? 64 : 32;      // words per row group per stage

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_a[s], 1);
      mbar_init(&full_b[s], kExp);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&acc_bar, 1);
    fail = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_base, kBN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  pdl_launch_dependents();
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp == 0) {
    if (lane == 0) {
      // Producer: TMA of the x_tilde tile [m0, m0+128) x [64 ks, 64 ks + 64)
      // and of the packed code words of the same 64 codes for the CTA's 16
      // row groups (one 2-D box of the tiled layout; rows past N read 0).
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
        if (!ok) break;
        const int cx = p.quantizer == SDQ_TERNARY ? (ks >> 1) * 128 + 64 * (ks & 1)
                                                   : (ks >> 2) * 128 + 32 * (ks & 3);
        mbar_expect_tx(&full_a[s], kATile + 16 * cwords * 4);
        tma_load_2d(a_tiles + s * kATile, &amap, ks * kBK, m0, &full_a[s]);
        tma_load_2d(base + kStages * (kATile + kBTile) + s * kCTile, &cmap, cx, n0 >> 4, &full_a[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        ok = mbar_wait(&full_a[s], r & 1) && mbar_wait(&full_b[s], r & 1);
        if (!ok) break;
        tc_fence_after();
        const uint64_t ad = sw128_desc(sbase + s * kATile);
        const uint64_t bd = sw128_desc(sbase + kStages * kATile + s * kBTile);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
          umma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, kIdesc, (ks | kk) != 0);
        umma_commit(&empty[s]);
      }
      umma_commit(&acc_bar);
    }
  } else {
    // B expanders: kExp threads.  Lane -> (g = lane % 8, t = lane / 8) so
    // the 8 lanes of each 128-bit store phase hit 8 distinct 16-byte banks.
    const int et = tid - 64;
    const int g = lane & 7, t = lane >> 3, L = 4 * g + t;
    for (int ks = 0; ks < p.nks && ok; ++ks) {
      const int s = ks % kStages, r = ks / kStages;
      if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
      if (ok) ok = mbar_wait(&full_a[s], r & 1);             // packed codes have landed
      if (!ok) break;
      uint8_t* bt = b_tiles + s * kBTile;
      const uint32_t* ct = c_tiles + s * (kCTile / 4);
      if (p.quantizer == SDQ_TERNARY) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int idx = (et >> 5) + 8 * u;            // (row group, word half) pair
          const int rgl = idx >> 1, qh = idx & 1;
          const uint32_t w = ct[rgl * 64 + 32 * qh + L];
          uint32_t v[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) v[j] = (w << (2 * j)) & 0xC000C000u;
          const int n = 16 * rgl + g, c8 = 4 * qh + t;
          st_chunk(bt, n, c8, v[0], v[2], v[4], v[6]);
          st_chunk(bt, n + 8, c8, v[1], v[3], v[5], v[7]);
        }
      } else {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int rgl = (et >> 5) + 8 * u;
          const uint32_t nw = ~ct[rgl * 32 + L];
          uint32_t v[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] = ((nw << j) & 0x80008000u) | 0x40004000u;
          const int n = 16 * rgl + g;
          st_chunk(bt, n, t, v[0], v[2], v[8], v[10]);
          st_chunk(bt, n, 4 + t, v[4], v[6], v[12], v[14]);
          st_chunk(bt, n + 8, t, v[1], v[3], v[9], v[11]);
          st_chunk(bt, n + 8, 4 + t, v[5], v[7], v[13], v[15]);
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&full_b[s]);
    }
    // Epilogue: TMEM quadrant (warp % 4) holds rows m0 + 32 (warp % 4) + lane.
    if (ok) ok = mbar_wait(&acc_bar, 0);
    tc_fence_after();
    if (ok) {
      const int qd = warp & 3;                       // TMEM lane quadrant of this warp
      const int half = (warp - 2) >> 2;              // warps 2..5 and 6..9 split the columns
      const int row = m0 + 32 * qd + lane;
      for (int cc = half * (kBN / 32); cc < (half + 1) * (kBN / 32); ++cc) {
        uint32_t r[16];
        tmem_ld16(tmem + ((uint32_t)(32 * qd) << 16) + 16 * cc, r);
        tmem_ld_wait();
        const int nb = n0 + 16 * cc;
        if (row < p.M) {
          float* yr = p.y + (size_t)row * p.N + nb;
          if (nb + 16 <= p.N && (p.N & 3) == 0) {
#pragma unroll
            for (int i = 0; i < 16; i += 4) {
              float4 v;
              v.x = __uint_as_float(r[i]) * 0.5f * __ldg(p.alpha + nb + i);
              v.y = __uint_as_float(r[i + 1]) * 0.5f * __ldg(p.alpha + nb + i + 1);
              v.z = __uint_as_float(r[i + 2]) * 0.5f * __ldg(p.alpha + nb + i + 2);
              v.w = __uint_as_float(r[i + 3]) * 0.5f * __ldg(p.alpha + nb + i + 3);
              *reinterpret_cast<float4*>(yr + i) = v;
            }
          } else {
            for (int i = 0; i < 16; ++i)
              if (nb + i < p.N) yr[i] = __uint_as_float(r[i]) * 0.5f * __ldg(p.alpha + nb + i);
          }
        }
      }
    }
  }
  if (!ok) {
    fail = 1;
    atomicExch(p.err, 1u);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kBN);
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

}  // namespace

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
  const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kBM};
  const cuuint32_t estr[2] = {1, 1};
  CUresult cr = enc(&amap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, wbase + L.xt, dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;
  // Tiled codes as a 2-D array: one row per row group, n_chunks * 128 words.
  CUtensorMap cmap;
  const cuuint64_t cdims[2] = {(cuuint64_t)g.n_chunks * 128, (cuuint64_t)g.ng};
  const cuuint64_t cstrides[1] = {(cuuint64_t)g.n_chunks * 512};
  const cuuint32_t cbox[2] = {(cuuint32_t)(pl->desc.quantizer == SDQ_TERNARY ? 64 : 32), 16};
  cr = enc(&cmap, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint32_t*>(codes), cdims, cstrides, cbox,
           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;
  PrefillParams p;
  p.codes = codes; p.alpha = alpha; p.y = y;
  p.err = reinterpret_cast<uint32_t*>(wbase + L.err);
  p.M = M; p.N = g.n_out; p.ng = g.ng; p.n_chunks = g.n_chunks;
  p.nks = (int)(g.k_eff_pad / kBK);
  p.quantizer = pl->desc.quantizer;
  cudaError_t e = cudaFuncSetAttribute(prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((g.n_out + kBN - 1) / kBN, (M + kBM - 1) / kBM);
  return launch_pdl(prefill_kernel, grid, dim3(kThreads), (size_t)kSmem, st, amap, cmap, p);
}

}  // namespace sdq
