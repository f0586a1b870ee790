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
// Output, decode path (M <= 64): fp32 x_tilde (M x K_eff_pad) plus, per CTA,
// max |x_tilde| for each batch row (the decode kernel turns these into the
// power-of-two scale of its fp8 expansion).  Prefill path: bf16 x_tilde in
// the permuted 64-code stage order of the prefill kernel's operand tiles.
#include "common.cuh"

namespace sdq {

namespace {

constexpr int kTile = 64;   // rows (blocks b) and columns (samples j) per CTA
constexpr int kKC = 32;     // k per smem stage
constexpr int kLd = kKC + 8;  // padded bf16 row stride

struct PrepParams {
  const uint16_t* x;
  const uint16_t* g_hi;
  const uint16_t* g_lo;
  float* xt;          // decode: fp32 M x kpad
  uint16_t* xtb;      // prefill: bf16 M x kpad (permuted)
  float* pmax;        // decode: M x P
  uint32_t* cnt;      // decode counters to zero
  int ncnt;
  int M, K, B, n_b, nblk, P, JT;
  int64_t k_eff, kpad;
  int prefill;
};

__global__ void __launch_bounds__(128) prep_kernel(PrepParams p) {
  __shared__ __align__(16) uint16_t xs[kTile * kLd];
  __shared__ __align__(16) uint16_t ghs[kTile * kLd];
  __shared__ __align__(16) uint16_t gls[kTile * kLd];
  __shared__ float red[4];
  const int jt = blockIdx.x, bt = blockIdx.y, m = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int b0 = bt * kTile, j0 = jt * kTile;

  float acc[8][4];
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[n][e] = 0.f;

  for (int kc = 0; kc < p.B; kc += kKC) {
    // Stage x rows (blocks) and G rows (samples), k in [kc, kc + 32).
    for (int i = tid; i < kTile * kKC; i += 128) {
      const int rr = i / kKC, kk = i - rr * kKC, k = kc + kk;
      const int b = b0 + rr, j = j0 + rr;
      xs[rr * kLd + kk] = (b < p.nblk && k < p.B) ? p.x[(size_t)m * p.K + (size_t)b * p.B + k] : 0;
      const bool gv = j < p.n_b && k < p.B;
      ghs[rr * kLd + kk] = gv ? p.g_hi[(size_t)j * p.B + k] : 0;
      gls[rr * kLd + kk] = gv ? p.g_lo[(size_t)j * p.B + k] : 0;
    }
    __syncthreads();
#pragma unroll
    for (int ks = 0; ks < kKC; ks += 16) {
      uint32_t a[4];
      const uint16_t* ar = xs + (warp * 16 + g) * kLd + ks + 2 * t;
      a[0] = *reinterpret_cast<const uint32_t*>(ar);
      a[1] = *reinterpret_cast<const uint32_t*>(ar + 8 * kLd);
      a[2] = *reinterpret_cast<const uint32_t*>(ar + 8);
      a[3] = *reinterpret_cast<const uint32_t*>(ar + 8 * kLd + 8);
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        const int off = (n * 8 + g) * kLd + ks + 2 * t;
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
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int b = b0 + warp * 16 + g + (e >> 1) * 8;
      const int j = j0 + n * 8 + 2 * t + (e & 1);
      if (b < p.nblk && j < p.n_b) {
        const int64_t kk = (int64_t)b * p.n_b + j;
        const float v = acc[n][e];
        if (p.prefill) {
          const int64_t phys = (kk & ~int64_t(63)) | prefill_perm64((int)(kk & 63));
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
        const int64_t phys = (k & ~int64_t(63)) | prefill_perm64((int)(k & 63));
        p.xtb[(size_t)m * p.kpad + phys] = 0;
      } else {
        p.xt[(size_t)m * p.kpad + k] = 0.f;
      }
    }
    if (m == 0 && p.cnt)
      for (int i = tid; i < p.ncnt; i += 128) p.cnt[i] = 0u;
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
  p.JT = (g.n_b + kTile - 1) / kTile;
  const int BT = (g.nblk + kTile - 1) / kTile;
  p.P = p.JT * BT;
  if (p.prefill) {
    p.pmax = nullptr; p.cnt = nullptr; p.ncnt = 0;
  } else {
    const DecodeConfig dc = decode_config(pl, M);
    p.pmax = reinterpret_cast<float*>(base + L.pmax);
    p.cnt = reinterpret_cast<uint32_t*>(base + L.cnt);
    p.ncnt = dc.R;
  }
  dim3 grid(p.JT, BT, M);
  prep_kernel<<<grid, 128, 0, st>>>(p);
  return cudaGetLastError();
}

}  // namespace sdq
