// K3: activation transform x_tilde = G x_b for every block b of B inputs.
//
// G = D^T Had^T (n_b x B) is the adjoint of the reconstruction of Algorithm 1
// (downsample the codes to B samples, undo the Hadamard smoothing), so that
// sum_j c[r,j] x_tilde[j] equals W_hat[r] . x exactly (section 3.5: the
// activations are upsampled with the layer's OSR).  Reshaping x (M x K) to
// (M*K/B) x B rows makes this one small GEMM against G^T, run on warp MMAs:
// x is bf16 (exact), G is split into bf16 hi + lo parts (relative error of
// the pair ~2^-16), accumulation in fp32.
//
// Decode path (M <= 64): fp32 x_tilde (M x K_eff_pad) plus max |x_tilde|
// per CTA and batch row; then the terms kernel below writes the decode
// kernel's e4m3 B operand.  Prefill path: bf16 x_tilde in the permuted
// 64-code stage order of the prefill kernel's operand tiles.
#include "common.cuh"

namespace sdq {

namespace {

constexpr int kKC = 32;       // k per smem stage
constexpr int kLd = kKC + 8;  // padded bf16 row stride

struct PrepParams {
  const uint16_t* x;
  const uint16_t* g_hi;
  const uint16_t* g_lo;
  float* xt;          // decode: fp32 M x kpad
  uint16_t* xtb;      // prefill: bf16 M x kpad (permuted)
  float* pmax;        // decode: M x P
  uint32_t* cnt;      // decode counters and error word to zero
  int ncnt;
  int M, K, B, n_b, nblk, P, JT;
  int64_t k_eff, kpad;
  int prefill, vec, ternary;
};

// CTA tile: TB blocks (rows) x 64 samples j, 4 warps.  TB = 64: each warp
// owns 16 rows x 64 j; TB = 16: each warp owns the 16 rows x 16 j.
template <int TB>
__global__ void __launch_bounds__(128) prep_kernel(PrepParams p) {
  constexpr int NTW = TB == 64 ? 8 : 2;   // 8-column MMA tiles per warp
  __shared__ __align__(16) uint16_t xs[TB * kLd];
  __shared__ __align__(16) uint16_t ghs[64 * kLd];
  __shared__ __align__(16) uint16_t gls[64 * kLd];
  __shared__ float red[4];
  pdl_wait();
  pdl_launch_dependents();
  const int jt = blockIdx.x, bt = blockIdx.y, m = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int b0 = bt * TB, j0 = jt * 64;
  const int wrow = TB == 64 ? warp * 16 : 0;       // warp's first row in the tile
  const int wcol = TB == 64 ? 0 : warp * 16;       // warp's first column

  float acc[NTW][4];
#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[n][e] = 0.f;

  for (int kc = 0; kc < p.B; kc += kKC) {
    if (p.vec) {  // 16-byte loads: B % 32 == 0, rows 16-byte aligned
      for (int i = tid; i < TB * 4; i += 128) {
        const int rr = i >> 2, q = i & 3, b = b0 + rr;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (b < p.nblk)
          v = *reinterpret_cast<const uint4*>(p.x + (size_t)m * p.K + (size_t)b * p.B + kc + 8 * q);
        *reinterpret_cast<uint4*>(xs + rr * kLd + 8 * q) = v;
      }
      for (int i = tid; i < 64 * 4; i += 128) {
        const int rr = i >> 2, q = i & 3, j = j0 + rr;
        uint4 vh = make_uint4(0, 0, 0, 0), vl = vh;
        if (j < p.n_b) {
          vh = *reinterpret_cast<const uint4*>(p.g_hi + (size_t)j * p.B + kc + 8 * q);
          vl = *reinterpret_cast<const uint4*>(p.g_lo + (size_t)j * p.B + kc + 8 * q);
        }
        *reinterpret_cast<uint4*>(ghs + rr * kLd + 8 * q) = vh;
        *reinterpret_cast<uint4*>(gls + rr * kLd + 8 * q) = vl;
      }
    } else {
      for (int i = tid; i < TB * kKC; i += 128) {
        const int rr = i / kKC, kk = i - rr * kKC, k = kc + kk, b = b0 + rr;
        xs[rr * kLd + kk] = (b < p.nblk && k < p.B) ? p.x[(size_t)m * p.K + (size_t)b * p.B + k] : 0;
      }
      for (int i = tid; i < 64 * kKC; i += 128) {
        const int rr = i / kKC, kk = i - rr * kKC, k = kc + kk, j = j0 + rr;
        const bool gv = j < p.n_b && k < p.B;
        ghs[rr * kLd + kk] = gv ? p.g_hi[(size_t)j * p.B + k] : 0;
        gls[rr * kLd + kk] = gv ? p.g_lo[(size_t)j * p.B + k] : 0;
      }
    }
    __syncthreads();
#pragma unroll
    for (int ks = 0; ks < kKC; ks += 16) {
      uint32_t a[4];
      const uint16_t* ar = xs + (wrow + g) * kLd + ks + 2 * t;
      a[0] = *reinterpret_cast<const uint32_t*>(ar);
      a[1] = *reinterpret_cast<const uint32_t*>(ar + 8 * kLd);
      a[2] = *reinterpret_cast<const uint32_t*>(ar + 8);
      a[3] = *reinterpret_cast<const uint32_t*>(ar + 8 * kLd + 8);
#pragma unroll
      for (int n = 0; n < NTW; ++n) {
        const int off = (wcol + n * 8 + g) * kLd + ks + 2 * t;
        const uint32_t h0 = *reinterpret_cast<const uint32_t*>(ghs + off);
        const uint32_t h1 = *reinterpret_cast<const uint32_t*>(ghs + off + 8);
        const uint32_t l0 = *reinterpret_cast<const uint32_t*>(gls + off);
        const uint32_t l1 = *reinterpret_cast<const uint32_t*>(gls + off + 8);
        mma_bf16_16816(acc[n], a, h0, h1);
        mma_bf16_16816(acc[n], a, l0, l1);
      }
    }
    __syncthreads();
  }

  float vmax = 0.f;
#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int b = b0 + wrow + g + (e >> 1) * 8;
      const int j = j0 + wcol + n * 8 + 2 * t + (e & 1);
      if (b < p.nblk && j < p.n_b) {
        const int64_t kk = (int64_t)b * p.n_b + j;
        const float v = acc[n][e];
        if (p.prefill) {
          const int64_t phys = (kk & ~int64_t(63)) | prefill_pos64((int)(kk & 63), p.ternary);
          p.xtb[(size_t)m * p.kpad + phys] = float_to_bf16_bits(v);
        } else {
          p.xt[(size_t)m * p.kpad + kk] = v;
          vmax = fmaxf(vmax, fabsf(v));
        }
      }
    }
  if (!p.prefill) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
    if (lane == 0) red[warp] = vmax;
    __syncthreads();
    if (tid == 0)
      p.pmax[(size_t)m * p.P + bt * p.JT + jt] = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
  }
  // Zero the K padding of this batch row, and the decode counters.
  if (jt == 0 && bt == 0) {
    for (int64_t k = p.k_eff + tid; k < p.kpad; k += 128) {
      if (p.prefill) {
        const int64_t phys = (k & ~int64_t(63)) | prefill_pos64((int)(k & 63), p.ternary);
        p.xtb[(size_t)m * p.kpad + phys] = 0;
      } else {
        p.xt[(size_t)m * p.kpad + k] = 0.f;
      }
    }
    if (m == 0 && p.cnt)
      for (int i = tid; i < p.ncnt; i += 128) p.cnt[i] = 0u;
  }
}

// ------------------------------------------------------------ e4m3 terms
// B operand of the decode MMAs for the whole K range: block kb (128 codes)
// is NP rows x 128 bytes in the 128-byte-swizzled K-major layout, row
// n = m T + t holding term t of batch row m at MMA K index kap (natural code
// decode_stage_k(kap)).  With e_m chosen so that max |x_tilde[m]| 2^-e_m <
// 448, v = x_tilde 2^-e_m splits into sum_t 16^-t q_t: q_t = e4m3(v_t),
// v_{t+1} = 16 (v_t - q_t) (exact: e4m3 rounding is relative, the residual
// has few bits).  Rows past M T are not written: they only feed
// accumulator columns that are never read.  One thread per (kb, m, 16-byte
// chunk); e_m also goes to sexp for the decode epilogue.
struct TermsParams {
  const float* xt;
  const float* pmax;
  uint8_t* bimg;
  int* sexp;
  int M, T, NP, pp, KB, ternary;
  int64_t kpad;
};

__global__ void __launch_bounds__(256) terms_kernel(TermsParams p) {
  __shared__ int se[kMaxDecodeM];
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x;
  if (tid < p.M) {
    float mx = 0.f;
    for (int i = 0; i < p.pp; ++i) mx = fmaxf(mx, p.pmax[(size_t)tid * p.pp + i]);
    int e = 0;
    if (mx > 0.f) frexpf(mx / 448.f, &e);   // max |x_tilde| * 2^-e < 448
    e = max(e, -120);
    se[tid] = e;
    if (blockIdx.x == 0) p.sexp[tid] = e;
  }
  __syncthreads();
  const int64_t it = (int64_t)blockIdx.x * blockDim.x + tid;
  if (it >= (int64_t)p.KB * p.M * 8) return;
  const int ch = (int)(it & 7);
  const int64_t mk = it >> 3;
  const int m = (int)(mk % p.M);
  const int64_t kb = mk / p.M;
  const float* xr = p.xt + (size_t)m * p.kpad + (size_t)kb * 128;
  const float inv = ldexpf(1.f, -se[m]);
  float v[16];
  if (p.ternary) {
    // K indices 16 ch .. 16 ch + 15 hold codes 16 ch .. 16 ch + 15, permuted
    const float4* x4 = reinterpret_cast<const float4*>(xr + 16 * ch);
    float xv[16];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = x4[q];
      xv[4 * q] = f.x; xv[4 * q + 1] = f.y; xv[4 * q + 2] = f.z; xv[4 * q + 3] = f.w;
    }
#pragma unroll
    for (int u = 0; u < 16; ++u) v[u] = xv[decode_stage_k(u, true)] * inv;
  } else {
#pragma unroll
    for (int u = 0; u < 16; ++u) v[u] = xr[decode_stage_k(16 * ch + u, false)] * inv;
  }
  uint8_t* dst = p.bimg + (size_t)kb * p.NP * 128;
  for (int t = 0; t < p.T; ++t) {
    uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const uint32_t q = f32_to_e4m3(v[u]);
      w[u >> 2] |= q << (8 * (u & 3));
      v[u] = (v[u] - e4m3_to_f32(q)) * 16.f;
    }
    const int n = m * p.T + t;
    *reinterpret_cast<uint4*>(dst + n * 128 + ((ch ^ (n & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

}  // namespace

cudaError_t launch_prep(const sdq_plan_s* pl, const uint16_t* x, int M, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  const WsLayout L = workspace_layout(pl, M);
  PrepParams p;
  p.x = x; p.g_hi = pl->d_g_hi; p.g_lo = pl->d_g_lo;
  uint8_t* base = static_cast<uint8_t*>(ws);
  p.prefill = M > kMaxDecodeM;
  p.xt = p.prefill ? nullptr : reinterpret_cast<float*>(base + L.xt);
  p.xtb = p.prefill ? reinterpret_cast<uint16_t*>(base + L.xt) : nullptr;
  p.M = M; p.K = g.k_in; p.B = g.block; p.n_b = g.n_b; p.nblk = g.nblk;
  p.k_eff = g.k_eff; p.kpad = g.k_eff_pad;
  p.ternary = pl->desc.quantizer == SDQ_TERNARY;
  p.vec = (g.block % 32 == 0) && ((reinterpret_cast<uintptr_t>(x) & 15u) == 0);
  const bool small = (int64_t)M * g.nblk < 4 * (int64_t)pl->sm_count;
  const int TB = small ? 16 : 64;
  p.JT = (g.n_b + 63) / 64;
  const int BT = (g.nblk + TB - 1) / TB;
  p.P = p.JT * BT;
  if (p.prefill) {
    p.pmax = nullptr;
    p.cnt = reinterpret_cast<uint32_t*>(base + L.err);   // the error word
    p.ncnt = 1;
  } else {
    p.pmax = reinterpret_cast<float*>(base + L.pmax);
    p.cnt = reinterpret_cast<uint32_t*>(base + L.cnt);
    p.ncnt = g.ntiles + 1;   // the tile tickets and the error word that follows them
  }
  dim3 grid(p.JT, BT, M);
  return small ? launch_pdl(prep_kernel<16>, grid, dim3(128), 0, st, p)
               : launch_pdl(prep_kernel<64>, grid, dim3(128), 0, st, p);
}

int prep_partials(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  const bool small = (int64_t)M * g.nblk < 4 * (int64_t)pl->sm_count;
  const int TB = small ? 16 : 64;
  return ((g.n_b + 63) / 64) * ((g.nblk + TB - 1) / TB);
}

cudaError_t launch_terms(const sdq_plan_s* pl, int M, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  const WsLayout L = workspace_layout(pl, M);
  const DecodeConfig& dc = decode_config(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  TermsParams p;
  p.xt = reinterpret_cast<const float*>(base + L.xt);
  p.pmax = reinterpret_cast<const float*>(base + L.pmax);
  p.bimg = base + L.bimg;
  p.sexp = reinterpret_cast<int*>(base + L.sexp);
  p.M = M; p.T = dc.T; p.NP = dc.NP; p.pp = dc.pp;
  p.KB = (int)(g.k_eff_pad / 128);
  p.ternary = g.bits == 2;
  p.kpad = g.k_eff_pad;
  const int64_t items = (int64_t)p.KB * M * 8;
  return launch_pdl(terms_kernel, dim3((unsigned)((items + 255) / 256)), dim3(256), 0, st, p);
}

}  // namespace sdq
