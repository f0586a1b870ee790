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
//   warp 0      TMEM allocation; lane 0 issues the TMA load of the A tile
//               and the bulk copies of the stage's two code slabs (tiled
//               layout: 128 rows x 64 codes each, contiguous)
//   warp 1      lane 0 issues tcgen05.mma (4 x K=16 per stage), commits to
//               the stage's "empty" barrier, finally to the accumulator one
//   warps 2..9  expand the B tile of every stage, one thread per code row:
//               the row's 64 codes (4 ternary / 2 binary words) become the
//               row's 128-byte line of bf16 (the shift-and-mask expansion
//               yields the codes in the permuted order the prep kernel also
//               uses for A), then read the fp32 accumulator out of TMEM
//               (tcgen05.ld), scale by alpha / 2 and store y.
// Every wait on an mbarrier is bounded (about 2 s); a timeout writes the call
// number into the workspace's call record and the CTA finishes without
// further waits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kATile = kBM * kBK * 2;     // 16 KB
constexpr int kBTile = kBN * kBK * 2;     // 32 KB
constexpr int kCTile = kBN * 16;          // packed codes of a stage: 2 slabs of up to 2 KB
constexpr int kSmem = kStages * (kATile + kBTile + kCTile) + 1024;
constexpr int kThreads = 320;   // 2 control warps + 8 expander / epilogue warps
constexpr int kExp = 256;       // expander threads

struct PrefillParams {
  const uint32_t* codes;
  const float* alpha;
  float* y;
  uint64_t* rec;       // call record
  uint64_t call;
  int M, N, ntiles, ngroups, wpg, nks, quantizer;
};

// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                            ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ void st_chunk(uint8_t* btile, int n, int c8, uint32_t a, uint32_t b,
                                         uint32_t c, uint32_t d) {
  uint4* p = reinterpret_cast<uint4*>(btile + n * 128 + ((c8 ^ (n & 7)) << 4));
  *p = make_uint4(a, b, c, d);
}

__global__ void __launch_bounds__(kThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap amap, PrefillParams p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_a[kStages], full_b[kStages], empty[kStages], acc_bar;
  __shared__ uint32_t tmem_base;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * kBN, m0 = blockIdx.y * kBM;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  uint8_t* base = smem_raw + (sbase - smem_u32(smem_raw));
  uint8_t* a_tiles = base;
  uint8_t* b_tiles = base + kStages * kATile;
  uint8_t* c_tiles = base + kStages * (kATile + kBTile);
  const uint32_t slab_bytes = (uint32_t)(kTileRows * p.wpg * 4);
  const int tile0 = blockIdx.x * (kBN / kTileRows);
  const int nslabs = min(kBN / kTileRows, p.ntiles - tile0);   // code slabs present per stage

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_a[s], 1);
      mbar_init(&full_b[s], kExp);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&acc_bar, 1);
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
  call_record_start(p.rec, p.call, blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0);
  const uint32_t tmem = tmem_base;
  bool ok = true;

  if (warp == 0) {
    if (lane == 0) {
      // Producer: TMA of the x_tilde tile [m0, m0+128) x [64 ks, 64 ks + 64)
      // and bulk copies of the code slabs (tile, group ks) of the CTA's
      // tiles (k group = stage: 64 codes).  A tile past the last one is not
      // copied; its rows are never stored.
      for (int ks = 0; ks < p.nks && ok; ++ks) {
        const int s = ks % kStages, r = ks / kStages;
        if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
        if (!ok) break;
        mbar_expect_tx(&full_a[s], kATile + nslabs * slab_bytes);
        tma_load_2d(a_tiles + s * kATile, &amap, ks * kBK, m0, &full_a[s]);
        for (int t = 0; t < nslabs; ++t) {
          const uint32_t* src = p.codes + (size_t)((int64_t)(tile0 + t) * p.ngroups + ks) * (slab_bytes / 4);
          bulk_g2s(c_tiles + s * kCTile + t * slab_bytes, src, slab_bytes, &full_a[s]);
        }
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
    // B expanders: thread et = code row n of the CTA tile (slab n / 128,
    // row n % 128).  Each thread writes its row's 128-byte line; the 8 lanes
    // of a 128-bit store phase hold 8 consecutive rows, whose swizzled chunk
    // positions differ, so the stores are free of bank conflicts.
    const int n = tid - 64;
    for (int ks = 0; ks < p.nks && ok; ++ks) {
      const int s = ks % kStages, r = ks / kStages;
      if (r > 0) ok = mbar_wait(&empty[s], (r - 1) & 1);
      if (ok) ok = mbar_wait(&full_a[s], r & 1);             // packed codes have landed
      if (!ok) break;
      uint8_t* bt = b_tiles + s * kBTile;
      const uint8_t* cs = c_tiles + s * kCTile + (n >> 7) * slab_bytes;
      if (p.quantizer == SDQ_TERNARY) {
        const uint4 w4 = *reinterpret_cast<const uint4*>(cs + (n & 127) * 16);
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          uint32_t v[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) v[j] = (w[i] << (2 * j)) & 0xC000C000u;
          st_chunk(bt, n, 2 * i, v[0], v[1], v[2], v[3]);
          st_chunk(bt, n, 2 * i + 1, v[4], v[5], v[6], v[7]);
        }
      } else {
        const uint2 w2 = *reinterpret_cast<const uint2*>(cs + (n & 127) * 8);
        const uint32_t w[2] = {~w2.x, ~w2.y};
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          uint32_t v[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] = ((w[i] << j) & 0x80008000u) | 0x40004000u;
#pragma unroll
          for (int c = 0; c < 4; ++c) st_chunk(bt, n, 4 * i + c, v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
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
  if (!ok) call_record_fail(p.rec, p.call);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();   // warp-collective: lane 0 ran the producer loop alone
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
  PrefillParams p;
  p.codes = codes; p.alpha = alpha; p.y = y;
  p.rec = reinterpret_cast<uint64_t*>(wbase + L.err);
  p.call = call_tag(next_call_number());
  p.M = M; p.N = g.n_out; p.ntiles = g.ntiles; p.ngroups = g.ngroups; p.wpg = g.wpg;
  p.nks = (int)(g.k_eff_pad / kBK);
  p.quantizer = pl->desc.quantizer;
  cudaError_t e = cudaFuncSetAttribute(prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((g.n_out + kBN - 1) / kBN, (M + kBM - 1) / kBM);
  return launch_pdl(prefill_kernel, grid, dim3(kThreads), (size_t)kSmem, st, amap, p);
}

}  // namespace sdq
