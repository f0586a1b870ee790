// K1: row-parallel Sigma-Delta encoder (SDQ-LLM Algorithm 1 without GPTQ
// compensation; eqs. (3)-(8)).
//
// One warp owns 4 output rows.  For every block of B input columns it
// rebuilds the upsampled block x_up = A_enc w (A_enc = U Had^T, the
// Hadamard smoothing of eq. (13) fused with the Resample upsampler) with all
// 32 lanes, each lane producing 4 of every 128 samples for the 4 rows, in
// the canonical fp32 order: one rounded product per term, k ascending, no
// FMA.  Pass 1 reduces alpha per row (exact max, or the sequential fp32
// mean); pass 2 recomputes x_up and lanes 0..3 run the first-order
// Sigma-Delta recursion of eq. (8) over their row, reset at every block, and
// write the codes in the plain packed layout.
#include "common.cuh"

namespace sdq {

namespace {

constexpr int kRW = 4;     // rows per warp
constexpr int kMaxWarps = 16;
constexpr int kJC = 128;   // upsampled samples per lane pass (4 per lane)

struct EncodeParams {
  const float* W;
  uint32_t* codes;
  float* alpha;
  const float* at;  // B x n_b, At[k][j] = A_enc[j][k]
  int n_out, k_in, B, n_b, nblk, wpr, quantizer, alpha_mode, warps;
  int64_t k_eff;
};

// kTable: the CTA first copies the table into shared memory (where it fits
// beside the warps' buffers); its reads in the product loop are then
// shared-memory hits instead of L2 round trips, on which the loop waited.
template <bool kTable>
__global__ void __launch_bounds__(32 * kMaxWarps) encode_kernel(EncodeParams p) {
  extern __shared__ float smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int xs_stride = p.n_b + 1;
  const float* at = p.at;
  float* wbuf = smem;
  if constexpr (kTable) {
    float* ts = smem;
    const int n = p.B * p.n_b;
    for (int i = threadIdx.x; i < n / 4; i += blockDim.x)
      reinterpret_cast<float4*>(ts)[i] = __ldg(reinterpret_cast<const float4*>(p.at) + i);
    __syncthreads();
    at = ts;
    wbuf = smem + n;
  }
  float* ws = wbuf + (size_t)warp * (kRW * p.B + kRW * xs_stride);
  float* xs = ws + kRW * p.B;
  const int row0 = (blockIdx.x * p.warps + warp) * kRW;
  if (row0 >= p.n_out) return;
  const int nrows = min(kRW, p.n_out - row0);
  const bool need_xs_pass0 = p.alpha_mode == SDQ_ALPHA_MEANABS;

  float amax[kRW];
#pragma unroll
  for (int r = 0; r < kRW; ++r) amax[r] = 0.f;
  float mean_acc = 0.f;  // lane r < 8: sequential sum for MEANABS
  bool mean_first = true;
  float alpha_row = 0.f;  // lane r < 8: alpha of row row0 + r

  for (int pass = 0; pass < 2; ++pass) {
    // pass-2 scan state of lane r (< nrows)
    uint32_t cw = 0;
    for (int b = 0; b < p.nblk; ++b) {
      __syncwarp();
      const float* wsrc = p.W + (size_t)row0 * p.k_in + (size_t)b * p.B;
      for (int i = lane; i < kRW * p.B; i += 32) {
        const int r = i / p.B, k = i - r * p.B;
        ws[i] = r < nrows ? __ldg(wsrc + (size_t)r * p.k_in + k) : 0.f;
      }
      __syncwarp();
      for (int jc = 0; jc < p.n_b; jc += kJC) {
        float acc[kRW][4];
        int jj[4];
        bool jv[4];
#pragma unroll
        for (int s = 0; s < 4; ++s) {
          jj[s] = jc + lane + 32 * s;
          jv[s] = jj[s] < p.n_b;
        }
        {
          float a[4];
#pragma unroll
          for (int s = 0; s < 4; ++s) a[s] = jv[s] ? at[jj[s]] : 0.f;
#pragma unroll
          for (int r = 0; r < kRW; ++r) {
            const float wk = ws[r * p.B];
#pragma unroll
            for (int s = 0; s < 4; ++s) acc[r][s] = __fmul_rn(a[s], wk);
          }
        }
        for (int k = 1; k < p.B; ++k) {
          float a[4];
#pragma unroll
          for (int s = 0; s < 4; ++s) a[s] = jv[s] ? at[(size_t)k * p.n_b + jj[s]] : 0.f;
#pragma unroll
          for (int r = 0; r < kRW; ++r) {
            const float wk = ws[r * p.B + k];
#pragma unroll
            for (int s = 0; s < 4; ++s) acc[r][s] = __fadd_rn(acc[r][s], __fmul_rn(a[s], wk));
          }
        }
        if (pass == 0 && !need_xs_pass0) {
#pragma unroll
          for (int r = 0; r < kRW; ++r)
#pragma unroll
            for (int s = 0; s < 4; ++s)
              if (jv[s]) amax[r] = fmaxf(amax[r], fabsf(acc[r][s]));
        } else {
#pragma unroll
          for (int r = 0; r < kRW; ++r)
#pragma unroll
            for (int s = 0; s < 4; ++s)
              if (jv[s]) xs[r * xs_stride + jj[s]] = acc[r][s];
        }
      }
      __syncwarp();
      if (pass == 0) {
        if (need_xs_pass0 && lane < nrows) {
          for (int j = 0; j < p.n_b; ++j) {
            const float v = fabsf(xs[lane * xs_stride + j]);
            mean_acc = mean_first ? v : __fadd_rn(mean_acc, v);
            mean_first = false;
          }
        }
      } else if (lane < nrows) {
        // Eq. (8): i = (i + x) - y_prev, reset per block.
        const float a = alpha_row, theta = 0.5f * alpha_row;
        float integ = 0.f, yp = 0.f;
        const int per = 32 / p.quantizer;
        uint32_t* crow = p.codes + (size_t)(row0 + lane) * p.wpr;
        for (int j = 0; j < p.n_b; ++j) {
          integ = __fsub_rn(__fadd_rn(integ, xs[lane * xs_stride + j]), yp);
          uint32_t field;
          if (p.quantizer == SDQ_TERNARY) {
            if (integ > theta) { field = 1u; yp = a; }
            else if (integ < -theta) { field = 3u; yp = -a; }
            else { field = 0u; yp = 0.f; }
          } else {
            if (integ >= 0.f) { field = 1u; yp = a; }
            else { field = 0u; yp = -a; }
          }
          const int64_t kk = (int64_t)b * p.n_b + j;
          const int pos = (int)(kk % per);
          cw |= field << (p.quantizer * pos);
          if (pos == per - 1 || kk == p.k_eff - 1) {
            crow[kk / per] = cw;
            cw = 0;
          }
        }
      }
    }
    if (pass == 0) {
      if (p.alpha_mode == SDQ_ALPHA_MAXABS) {
#pragma unroll
        for (int r = 0; r < kRW; ++r) {
          float v = amax[r];
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
          if (lane == r) alpha_row = v;
        }
      } else if (lane < nrows) {
        alpha_row = __fdiv_rn(mean_acc, (float)p.k_eff);
      }
      if (lane < nrows) p.alpha[row0 + lane] = alpha_row;
    }
  }
  // Zero the row padding words past the last code.
  if (lane < nrows) {
    const int per = 32 / p.quantizer;
    uint32_t* crow = p.codes + (size_t)(row0 + lane) * p.wpr;
    for (int64_t w = (p.k_eff + per - 1) / per; w < p.wpr; ++w) crow[w] = 0u;
  }
}

}  // namespace

cudaError_t launch_encode(const sdq_plan_s* pl, const float* W, uint32_t* codes, float* alpha,
                          cudaStream_t st) {
  const Geometry& g = pl->geo;
  EncodeParams p;
  p.W = W; p.codes = codes; p.alpha = alpha; p.at = pl->d_at;
  p.n_out = g.n_out; p.k_in = g.k_in; p.B = g.block; p.n_b = g.n_b; p.nblk = g.nblk;
  p.wpr = g.words_per_row; p.quantizer = pl->desc.quantizer; p.alpha_mode = pl->desc.alpha_mode;
  p.k_eff = g.k_eff;
  const size_t per_warp = sizeof(float) * ((size_t)kRW * g.block + (size_t)kRW * (g.n_b + 1));
  const size_t table = sizeof(float) * (size_t)g.block * g.n_b;
  if (per_warp > 227 * 1024) return cudaErrorInvalidConfiguration;
  // the table in shared memory when it fits beside at least 4 warps' buffers
  // (a multiple of 4 floats: copied as float4)
  const bool in_smem = (g.block * g.n_b) % 4 == 0 && table + 4 * per_warp <= 224 * 1024;
  int warps = (int)(((in_smem ? 224 * 1024 - table : 200 * 1024)) / per_warp);
  warps = warps < 1 ? 1 : (warps > kMaxWarps ? kMaxWarps : warps);
  p.warps = warps;
  const size_t smem = per_warp * warps + (in_smem ? table : 0);
  cudaError_t e = in_smem ? cudaFuncSetAttribute(encode_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem)
                          : cudaFuncSetAttribute(encode_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
  if (e != cudaSuccess) return e;
  const int rows_per_cta = warps * kRW;
  const int grid = (g.n_out + rows_per_cta - 1) / rows_per_cta;
  if (in_smem) encode_kernel<true><<<grid, warps * 32, smem, st>>>(p);
  else encode_kernel<false><<<grid, warps * 32, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace sdq
