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
// Decode path (M <= 64): the decode prepare kernel below (x_tilde and the
// decode kernel's e4m3 B operand in one pass).  Prefill path: bf16 x_tilde
// in the permuted 64-code stage order of the prefill kernel's operand tiles.
#include <algorithm>

#include "common.cuh"

namespace sdq {

namespace {

constexpr int kKC = 32;       // k per smem stage
constexpr int kLd = kKC + 8;  // padded bf16 row stride

// Prefill prepare (M > 64): bf16 x_tilde, each 64-code stage of K in the
// prefill kernel's operand order (prefill_pos64).
struct PrepParams {
  const uint16_t* x;
  const uint16_t* g_hi;
  const uint16_t* g_lo;
  uint16_t* xtb;      // bf16 M x kpad (permuted)
  int M, K, B, n_b, nblk;
  int64_t k_eff, kpad;
  int vec, ternary;
};

// CTA tile: TB blocks (rows) x 64 samples j, 4 warps.  TB = 64: each warp
// owns 16 rows x 64 j; TB = 16: each warp owns the 16 rows x 16 j.
template <int TB>
__global__ void __launch_bounds__(128) prep_kernel(PrepParams p) {
  constexpr int NTW = TB == 64 ? 8 : 2;   // 8-column MMA tiles per warp
  __shared__ __align__(16) uint16_t xs[TB * kLd];
  __shared__ __align__(16) uint16_t ghs[64 * kLd];
  __shared__ __align__(16) uint16_t gls[64 * kLd];
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

#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int b = b0 + wrow + g + (e >> 1) * 8;
      const int j = j0 + wcol + n * 8 + 2 * t + (e & 1);
      if (b < p.nblk && j < p.n_b) {
        const int64_t kk = (int64_t)b * p.n_b + j;
        const int64_t phys = (kk & ~int64_t(63)) | prefill_pos64((int)(kk & 63), p.ternary);
        p.xtb[(size_t)m * p.kpad + phys] = float_to_bf16_bits(acc[n][e]);
      }
    }
  // Zero the K padding of this batch row.
  if (jt == 0 && bt == 0) {
    for (int64_t k = p.k_eff + tid; k < p.kpad; k += 128) {
      const int64_t phys = (k & ~int64_t(63)) | prefill_pos64((int)(k & 63), p.ternary);
      p.xtb[(size_t)m * p.kpad + phys] = 0;
    }
  }
}

// ------------------------------------------------- decode prepare (M <= 64)
// One kernel per call: x_tilde = G x_b as above (fp32, kept for checking),
// and directly the decode kernel's e4m3 B operand.  That operand covers all
// of K: block kb (128 codes) is NP rows x 128 bytes in the 128-byte-swizzled
// K-major layout, row n = m T + t holding term t of batch row m at the MMA K
// position of each code (decode_pos).  With x_tilde[m] 2^-e_m < 448,
// v = x_tilde 2^-e_m splits into sum_t 16^-t q_t: q_t = e4m3(v_t),
// v_{t+1} = 16 (v_t - q_t) (exact: e4m3 rounding is relative).  e_m comes
// from a bound rather than from the maximum of x_tilde, so that no CTA waits
// for another: |x_tilde[m, j]| <= sum_k |G[j, k]| |x[m, k]| <= gnorm max|x[m]|,
// gnorm = max_j sum_k |G[j, k]| (with a margin for the bf16 split of G).
// e4m3 is floating point, so the looser scale costs no relative precision.
// Rows past M T are not written: they only feed accumulator columns that
// are never read.  The CTA's x tile and G rows arrive in one round of loads
// (k chunks of up to 256), overlapped with its reading of the x row for
// max |x[m]|.
struct DecPrepParams {
  const uint16_t* x;
  const uint16_t* g_hi;
  const uint16_t* g_lo;
  float* xt;          // M x kpad fp32
  uint8_t* bimg;      // e4m3 B operand image
  int* sexp;          // e_m per batch row
  float gnorm;
  int M, K, B, n_b, nblk, T, NP, kc, ternary, vec;
  int64_t k_eff, kpad;
};

__device__ __forceinline__ float bf16_abs(uint32_t h) { return __uint_as_float((h & 0x7FFFu) << 16); }

// 16-byte global -> shared copy that does not pass through registers; `bytes`
// = 0 fills the destination with zeros.
__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n"
               :: "r"(smem_u32(dst)), "l"(src), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;\n" ::: "memory");
}

__global__ void __launch_bounds__(128) prep_decode_kernel(DecPrepParams p) {
  constexpr int TB = 16, NTW = 2;   // 16 blocks x 64 j per CTA; warp w owns j 16w .. 16w + 15
  extern __shared__ __align__(16) uint8_t dsm[];
  const int ld = p.kc + 8;
  uint16_t* xs = reinterpret_cast<uint16_t*>(dsm);   // TB x ld
  uint16_t* ghs = xs + TB * ld;                        // 64 x ld
  uint16_t* gls = ghs + 64 * ld;                       // 64 x ld
  __shared__ float red[4];
  __shared__ int e_s;
  pdl_wait();
  pdl_launch_dependents();
  const int jt = blockIdx.x, bt = blockIdx.y, m = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int b0 = bt * TB, j0 = jt * 64, wcol = warp * 16;
  const uint16_t* xr = p.x + (size_t)m * p.K;

  float acc[NTW][4];
#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[n][e] = 0.f;
  float xmax = 0.f;
  for (int kc0 = 0; kc0 < p.B; kc0 += p.kc) {
    if (p.vec) {   // B % 32 == 0, rows 16-byte aligned: asynchronous 16-byte copies
      const int q8 = p.kc / 8;
      for (int i = tid; i < TB * q8; i += 128) {
        const int rr = i / q8, q = i - rr * q8, b = b0 + rr;
        const bool v = b < p.nblk;
        cp_async16(xs + rr * ld + 8 * q, v ? xr + (size_t)b * p.B + kc0 + 8 * q : xr, v ? 16u : 0u);
      }
      for (int i = tid; i < 64 * q8; i += 128) {
        const int rr = i / q8, q = i - rr * q8, j = j0 + rr;
        const bool v = j < p.n_b;
        const size_t off = v ? (size_t)j * p.B + kc0 + 8 * q : 0;
        cp_async16(ghs + rr * ld + 8 * q, p.g_hi + off, v ? 16u : 0u);
        cp_async16(gls + rr * ld + 8 * q, p.g_lo + off, v ? 16u : 0u);
      }
    } else {
      for (int i = tid; i < TB * p.kc; i += 128) {
        const int rr = i / p.kc, kk = i - rr * p.kc, k = kc0 + kk, b = b0 + rr;
        xs[rr * ld + kk] = (b < p.nblk && k < p.B) ? xr[(size_t)b * p.B + k] : 0;
      }
      for (int i = tid; i < 64 * p.kc; i += 128) {
        const int rr = i / p.kc, kk = i - rr * p.kc, k = kc0 + kk, j = j0 + rr;
        const bool gv = j < p.n_b && k < p.B;
        ghs[rr * ld + kk] = gv ? p.g_hi[(size_t)j * p.B + k] : 0;
        gls[rr * ld + kk] = gv ? p.g_lo[(size_t)j * p.B + k] : 0;
      }
    }
    if (kc0 == 0) {
      // max |x[m, :]| while the tile copies are in flight; 8 independent
      // 16-byte loads per thread at a time.
      if (p.vec) {
        const int nv = p.K / 8;
        for (int i0 = tid; i0 < nv; i0 += 128 * 8) {
          uint4 v[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int i = i0 + 128 * u;
            v[u] = i < nv ? __ldg(reinterpret_cast<const uint4*>(xr) + i) : make_uint4(0, 0, 0, 0);
          }
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) xmax = fmaxf(xmax, fmaxf(bf16_abs(w[q]), bf16_abs(w[q] >> 16)));
          }
        }
      } else {
        for (int i = tid; i < p.K; i += 128) xmax = fmaxf(xmax, bf16_abs(xr[i]));
      }
    }
    if (p.vec) cp_async_wait_all();
    __syncthreads();
    for (int ks = 0; ks < p.kc; ks += 16) {
      uint32_t a[4];
      const uint16_t* ar = xs + g * ld + ks + 2 * t;
      a[0] = *reinterpret_cast<const uint32_t*>(ar);
      a[1] = *reinterpret_cast<const uint32_t*>(ar + 8 * ld);
      a[2] = *reinterpret_cast<const uint32_t*>(ar + 8);
      a[3] = *reinterpret_cast<const uint32_t*>(ar + 8 * ld + 8);
#pragma unroll
      for (int n = 0; n < NTW; ++n) {
        const int off = (wcol + n * 8 + g) * ld + ks + 2 * t;
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

  // term scale exponent e_m from the bound
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) xmax = fmaxf(xmax, __shfl_xor_sync(0xffffffffu, xmax, o));
  if (lane == 0) red[warp] = xmax;
  __syncthreads();
  if (tid == 0) {
    const float mx = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
    int e = 0;
    if (mx > 0.f) {   // bound = mx gnorm < 2^(e1 + e2) without forming it (no overflow)
      int e1 = 0, e2 = 0;
      frexpf(mx, &e1);
      frexpf(p.gnorm, &e2);
      e = e1 + e2 - 8;   // bound * 2^-e < 256 < 448
    }
    e = max(e, -120);
    e_s = e;
    if (jt == 0 && bt == 0) p.sexp[m] = e;
  }
  __syncthreads();
  const float inv = ldexpf(1.f, -e_s);
  const bool ter = p.ternary != 0;
#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int b = b0 + g + (e >> 1) * 8;
      const int j = j0 + wcol + n * 8 + 2 * t + (e & 1);
      if (b < p.nblk && j < p.n_b) {
        const int64_t kk = (int64_t)b * p.n_b + j;
        p.xt[(size_t)m * p.kpad + kk] = acc[n][e];
        uint8_t* blk = p.bimg + (size_t)(kk >> 7) * p.NP * 128;
        const int kap = decode_pos((int)(kk & 127), ter);
        float v = acc[n][e] * inv;
        for (int tt = 0; tt < p.T; ++tt) {
          const uint32_t q = f32_to_e4m3(v);
          const int row = m * p.T + tt;
          blk[row * 128 + (((kap >> 4) ^ (row & 7)) << 4) + (kap & 15)] = (uint8_t)q;
          v = (v - e4m3_to_f32(q)) * 16.f;
        }
      }
    }
  // K padding of this batch row (x_tilde and its terms are 0 there).
  if (jt == 0 && bt == 0) {
    for (int64_t k = p.k_eff + tid; k < p.kpad; k += 128) {
      p.xt[(size_t)m * p.kpad + k] = 0.f;
      uint8_t* blk = p.bimg + (size_t)(k >> 7) * p.NP * 128;
      const int kap = decode_pos((int)(k & 127), ter);
      for (int tt = 0; tt < p.T; ++tt) {
        const int row = m * p.T + tt;
        blk[row * 128 + (((kap >> 4) ^ (row & 7)) << 4) + (kap & 15)] = 0;
      }
    }
  }
}

}  // namespace

cudaError_t launch_prep(const sdq_plan_s* pl, const uint16_t* x, int M, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  const int vec = (g.block % 32 == 0) && ((reinterpret_cast<uintptr_t>(x) & 15u) == 0);
  if (M <= kMaxDecodeM) {
    const DecodeConfig& dc = decode_config(pl, M);
    DecPrepParams p;
    p.x = x; p.g_hi = pl->d_g_hi; p.g_lo = pl->d_g_lo;
    p.xt = reinterpret_cast<float*>(base + L.xt);
    p.bimg = base + L.bimg;
    p.sexp = reinterpret_cast<int*>(base + L.sexp);
    p.gnorm = pl->gnorm;
    p.M = M; p.K = g.k_in; p.B = g.block; p.n_b = g.n_b; p.nblk = g.nblk;
    p.T = dc.T; p.NP = dc.NP;
    p.kc = std::max(16, std::min(g.block, 256));
    p.ternary = g.bits == 2;
    p.vec = vec;
    p.k_eff = g.k_eff; p.kpad = g.k_eff_pad;
    const size_t smem = (size_t)(16 + 128) * (p.kc + 8) * sizeof(uint16_t);
    static std::atomic<int> smem_set[64];   // per device: limit raised to the largest kc's need
    cudaError_t e = smem_limit_once(prep_decode_kernel, (16 + 128) * (256 + 8) * (int)sizeof(uint16_t),
                                    pl->device, smem_set);
    if (e != cudaSuccess) return e;
    dim3 grid((g.n_b + 63) / 64, (g.nblk + 15) / 16, M);
    return launch_pdl(prep_decode_kernel, grid, dim3(128), smem, st, p);
  }
  PrepParams p;
  p.x = x; p.g_hi = pl->d_g_hi; p.g_lo = pl->d_g_lo;
  p.xtb = reinterpret_cast<uint16_t*>(base + L.xt);
  p.M = M; p.K = g.k_in; p.B = g.block; p.n_b = g.n_b; p.nblk = g.nblk;
  p.k_eff = g.k_eff; p.kpad = g.k_eff_pad;
  p.ternary = pl->desc.quantizer == SDQ_TERNARY;
  p.vec = vec;
  const bool small = (int64_t)M * g.nblk < 4 * (int64_t)pl->sm_count;
  const int TB = small ? 16 : 64;
  dim3 grid((g.n_b + 63) / 64, (g.nblk + TB - 1) / TB, M);
  return small ? launch_pdl(prep_kernel<16>, grid, dim3(128), 0, st, p)
               : launch_pdl(prep_kernel<64>, grid, dim3(128), 0, st, p);
}

}  // namespace sdq
