// K1: row-parallel Sigma-Delta encoder (SDQ-LLM Algorithm 1, eqs. (3)-(8)),
// and the per-block half of its GPTQ compensation.
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
//
// The kernel covers a range of passes and blocks.  The encoder with GPTQ
// block compensation (Algorithm 1's outer loop with the inverse Hessian)
// runs pass 1 one block at a time on a working copy of W: after the scan,
// the warp rebuilds the block Q = alpha (c . G), forms E = W_F - Q and the
// normalised error E~ = E U_FF^-1 (forward substitution over the block's
// columns), which gptq_update_kernel then applies to the later columns.
#include "encode.cuh"

namespace sdq {

namespace {

constexpr int kRW = 4;     // rows per warp
constexpr int kMaxWarps = 16;
constexpr int kJC = 128;   // upsampled samples per lane pass (4 per lane)

struct EncodeParams {
  const float* W;
  uint32_t* codes;
  float* alpha;       // written by pass 0, read by pass 1 when pass 0 is not run
  const float* at;  // B x n_b, At[k][j] = A_enc[j][k]
  int n_out, k_in, B, n_b, nblk, wpr, quantizer, alpha_mode, warps;
  int64_t k_eff;
  int pass0, pass1, b0, b1;  // passes [pass0, pass1), blocks [b0, b1)
  // GPTQ (et non-null): G in fp32 (n_b x B), the factor U (k_in x k_in,
  // upper), and the normalised block error E~ written per row (n_out x B)
  const float* g32;
  const float* U;
  float* et;
};

// The warp's GPTQ step for block b of its rows, after the scan: xs holds the
// rows' codes (as +-1 / 0 floats), ws the block's current weights.  In the
// order of the oracle's canonical definition: s_k = sum_j c_j G[j][k] from
// +0 in ascending j, E_k = W_k - alpha s_k; then for l ascending E~_l =
// t_l / U_ll and t_k -= E~_l U_lk for k > l (t starts as E).  Lane owns
// columns k = lane (mod 32); t and E~ live in ws in place.
__device__ __noinline__ void gptq_block_error(const EncodeParams p, int b, int row0, int nrows, float* ws,
                                              const float* xs, int xs_stride, float alpha_row) {
  const int lane = threadIdx.x & 31;
  float ar[kRW];
#pragma unroll
  for (int r = 0; r < kRW; ++r) ar[r] = __shfl_sync(0xffffffffu, alpha_row, r);
  __syncwarp();
  // 128 columns at a time (4 per lane), j outermost: every (row, column) sum
  // still runs over j in ascending order, with 16 independent sums per lane
  for (int kc = 0; kc < p.B; kc += 128) {
    float sacc[kRW][4];
#pragma unroll
    for (int r = 0; r < kRW; ++r)
#pragma unroll
      for (int q = 0; q < 4; ++q) sacc[r][q] = 0.f;
    for (int j = 0; j < p.n_b; ++j) {
      float gv[4], xv[kRW];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int k = kc + lane + 32 * q;
        gv[q] = k < p.B ? __ldg(p.g32 + (size_t)j * p.B + k) : 0.f;
      }
#pragma unroll
      for (int r = 0; r < kRW; ++r) xv[r] = xs[r * xs_stride + j];
#pragma unroll
      for (int r = 0; r < kRW; ++r)
#pragma unroll
        for (int q = 0; q < 4; ++q) sacc[r][q] = __fadd_rn(sacc[r][q], __fmul_rn(xv[r], gv[q]));
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int k = kc + lane + 32 * q;
      if (k >= p.B) continue;
#pragma unroll
      for (int r = 0; r < kRW; ++r) ws[r * p.B + k] = __fsub_rn(ws[r * p.B + k], __fmul_rn(ar[r], sacc[r][q]));
    }
  }
  const size_t ldu = (size_t)p.k_in;
  const float* uff = p.U + (size_t)b * p.B * ldu + (size_t)b * p.B;
  for (int l = 0; l < p.B; ++l) {
    __syncwarp();
    const float d = __ldg(uff + (size_t)l * ldu + l);
    float el[kRW];
#pragma unroll
    for (int r = 0; r < kRW; ++r) el[r] = __fdiv_rn(ws[r * p.B + l], d);
    __syncwarp();
    if ((l & 31) == lane) {
#pragma unroll
      for (int r = 0; r < kRW; ++r) ws[r * p.B + l] = el[r];
    }
    for (int k = lane; k < p.B; k += 32) {
      if (k <= l) continue;
      const float u = __ldg(uff + (size_t)l * ldu + k);
#pragma unroll
      for (int r = 0; r < kRW; ++r) ws[r * p.B + k] = __fsub_rn(ws[r * p.B + k], __fmul_rn(el[r], u));
    }
  }
  __syncwarp();
  for (int i = lane; i < nrows * p.B; i += 32) {
    const int r = i / p.B, k = i - r * p.B;
    p.et[(size_t)(row0 + r) * p.B + k] = ws[i];
  }
  __syncwarp();
}

// kTable: the CTA first copies the table into shared memory (where it fits
// beside the warps' buffers); its reads in the product loop are then
// shared-memory hits instead of L2 round trips, on which the loop waited.
template <bool kTable, bool kGptq>
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
  if (p.pass0 == 1 && lane < nrows) alpha_row = p.alpha[row0 + lane];
  const int per = 32 / p.quantizer;

  for (int pass = p.pass0; pass < p.pass1; ++pass) {
    // pass-2 scan state of lane r (< nrows): the partial code word; a range
    // that starts inside a word continues the word its predecessor wrote
    uint32_t cw = 0;
    if (pass == 1 && lane < nrows && ((int64_t)p.b0 * p.n_b) % per != 0)
      cw = p.codes[(size_t)(row0 + lane) * p.wpr + (int64_t)p.b0 * p.n_b / per];
    for (int b = p.b0; b < p.b1; ++b) {
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
        uint32_t* crow = p.codes + (size_t)(row0 + lane) * p.wpr;
        const bool range_end = b == p.b1 - 1;
        for (int j = 0; j < p.n_b; ++j) {
          integ = __fsub_rn(__fadd_rn(integ, xs[lane * xs_stride + j]), yp);
          uint32_t field;
          float cv;
          if (p.quantizer == SDQ_TERNARY) {
            if (integ > theta) { field = 1u; yp = a; cv = 1.f; }
            else if (integ < -theta) { field = 3u; yp = -a; cv = -1.f; }
            else { field = 0u; yp = 0.f; cv = 0.f; }
          } else {
            if (integ >= 0.f) { field = 1u; yp = a; cv = 1.f; }
            else { field = 0u; yp = -a; cv = -1.f; }
          }
          if (kGptq) xs[lane * xs_stride + j] = cv;
          const int64_t kk = (int64_t)b * p.n_b + j;
          const int pos = (int)(kk % per);
          cw |= field << (p.quantizer * pos);
          if (pos == per - 1 || kk == p.k_eff - 1 || (range_end && j == p.n_b - 1)) {
            crow[kk / per] = cw;
            cw = 0;
          }
        }
      }
      if (kGptq && pass == 1) gptq_block_error(p, b, row0, nrows, ws, xs, xs_stride, alpha_row);
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
  if (p.pass1 == 2 && p.b1 == p.nblk && lane < nrows) {
    uint32_t* crow = p.codes + (size_t)(row0 + lane) * p.wpr;
    for (int64_t w = (p.k_eff + per - 1) / per; w < p.wpr; ++w) crow[w] = 0u;
  }
}

}  // namespace

cudaError_t launch_encode(const sdq_plan_s* pl, const float* W, uint32_t* codes, float* alpha,
                          cudaStream_t st) {
  return launch_encode_range(pl, W, codes, alpha, st, 0, 2, 0, pl->geo.nblk, nullptr, nullptr);
}

cudaError_t launch_encode_range(const sdq_plan_s* pl, const float* W, uint32_t* codes, float* alpha,
                                cudaStream_t st, int pass0, int pass1, int b0, int b1, const float* U,
                                float* et) {
  const Geometry& g = pl->geo;
  EncodeParams p;
  p.W = W; p.codes = codes; p.alpha = alpha; p.at = pl->d_at;
  p.n_out = g.n_out; p.k_in = g.k_in; p.B = g.block; p.n_b = g.n_b; p.nblk = g.nblk;
  p.wpr = g.words_per_row; p.quantizer = pl->desc.quantizer; p.alpha_mode = pl->desc.alpha_mode;
  p.k_eff = g.k_eff;
  p.pass0 = pass0; p.pass1 = pass1; p.b0 = b0; p.b1 = b1;
  p.g32 = pl->d_g32; p.U = U; p.et = et;
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
  const bool gptq = et != nullptr;
  auto kern = in_smem ? (gptq ? encode_kernel<true, true> : encode_kernel<true, false>)
                      : (gptq ? encode_kernel<false, true> : encode_kernel<false, false>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int rows_per_cta = warps * kRW;
  const int grid = (g.n_out + rows_per_cta - 1) / rows_per_cta;
  kern<<<grid, warps * 32, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace sdq
