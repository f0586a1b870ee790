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
// Decode path (M <= 64): the decode prepare kernel below writes fp32
// x_tilde, from which each decode CTA forms the e2m1 terms and scales of its
// k chunk.  Prefill path: bf16 x_tilde in the permuted 64-code stage order
// of the prefill kernel's operand tiles.
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
// One kernel per call: x_tilde = G x_b as above, fp32, M x kpad (the K
// padding zeroed), and, when n_b is a multiple of 64 (`bimg` set), the
// decode kernel's B operand for all of K: per 32-code group g of batch row
// m the power of two 2^e with |x_tilde 2^-e| < 4 (from the group's maximum)
// and T e2m1 terms, x_tilde = sum_t 2^(e - 3t) q_t, each term the 8x-scaled
// rounding error of the ones before.  Term t of row m is image row
// n = m T + t: 128-code block kb occupies bytes 64 (kb & 1) .. + 63 of the
// 128-byte rows of atom kb / 2 (NP rows, 128-byte swizzle), MMA position
// kap = 2 byte + nibble (decode_pos order); its scales are the bytes of
// word (kb, n) of `sfbw`: byte 2 mu + beta = 2^(e - 3t) of K group beta of
// the block's MMA mu.  The CTA's x tile and G rows arrive in one round of
// asynchronous copies (k chunks of up to 256).
struct DecPrepParams {
  const uint16_t* x;
  const uint16_t* g_hi;
  const uint16_t* g_lo;
  float* xt;          // M x kpad fp32
  uint8_t* bimg;      // B operand image (null: x_tilde only)
  uint8_t* sfbw;      // B scale words, KB x NP x 4 bytes
  float* y_zero;      // cleared (M x n_out) for the decode kernel's atomic split-K, or null
  int64_t y_count;
  int M, K, B, n_b, nblk, kc, vec, T, NP, ternary;
  int64_t k_eff, kpad;
};

__global__ void __launch_bounds__(128) prep_decode_kernel(DecPrepParams p) {
  constexpr int TB = 16, NTW = 2;   // 16 blocks x 64 j per CTA; warp w owns j 16w .. 16w + 15
  extern __shared__ __align__(16) uint8_t dsm[];
  const int ld = p.kc + 8;
  uint16_t* xs = reinterpret_cast<uint16_t*>(dsm);   // TB x ld
  uint16_t* ghs = xs + TB * ld;                        // 64 x ld
  uint16_t* gls = ghs + 64 * ld;                       // 64 x ld
  // The decode kernel may start right away: it waits for this grid to
  // complete before it reads anything this grid writes (y, the workspace).
  pdl_launch_dependents();
  const int jt = blockIdx.x, bt = blockIdx.y, m = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int b0 = bt * TB, j0 = jt * 64, wcol = warp * 16;
  const uint16_t* xr = p.x + (size_t)m * p.K;
  // G's rows for the first k chunk before waiting for the preceding grid: the
  // plan's tables are never written by the stream
  auto load_g = [&](int kc0) {
    const int q8 = p.kc / 8;
    for (int i = tid; i < 64 * q8; i += 128) {
      const int rr = i / q8, q = i - rr * q8, j = j0 + rr;
      const bool v = j < p.n_b;
      const size_t off = v ? (size_t)j * p.B + kc0 + 8 * q : 0;
      cp_async16(ghs + rr * ld + 8 * q, p.g_hi + off, v ? 16u : 0u);
      cp_async16(gls + rr * ld + 8 * q, p.g_lo + off, v ? 16u : 0u);
    }
  };
  if (p.vec) load_g(0);
  pdl_wait();
  if (p.y_zero) {   // grid-stride clear of y
    const int64_t nthr = (int64_t)gridDim.x * gridDim.y * gridDim.z * 128;
    const int64_t i0 = ((int64_t)(blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x) * 128 + tid;
    for (int64_t i = i0; i < p.y_count; i += nthr) p.y_zero[i] = 0.f;
  }

  float acc[NTW][4];
#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[n][e] = 0.f;
  for (int kc0 = 0; kc0 < p.B; kc0 += p.kc) {
    if (p.vec) {   // B % 32 == 0, rows 16-byte aligned: asynchronous 16-byte copies
      const int q8 = p.kc / 8;
      for (int i = tid; i < TB * q8; i += 128) {
        const int rr = i / q8, q = i - rr * q8, b = b0 + rr;
        const bool v = b < p.nblk;
        cp_async16(xs + rr * ld + 8 * q, v ? xr + (size_t)b * p.B + kc0 + 8 * q : xr, v ? 16u : 0u);
      }
      if (kc0 > 0) load_g(kc0);
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

  // x_tilde of the tile: to global memory (fp32) and to shared memory (the G
  // tiles are no longer read) for the terms below
  float* tile = reinterpret_cast<float*>(dsm);   // TB x 64
#pragma unroll
  for (int n = 0; n < NTW; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int bl = g + (e >> 1) * 8, jl = wcol + n * 8 + 2 * t + (e & 1);
      const int b = b0 + bl, j = j0 + jl;
      if (b < p.nblk && j < p.n_b) p.xt[(size_t)m * p.kpad + (int64_t)b * p.n_b + j] = acc[n][e];
      tile[bl * 64 + jl] = acc[n][e];
    }
  // K padding of this batch row
  if (jt == 0 && bt == 0)
    for (int64_t k = p.k_eff + tid; k < p.kpad; k += 128) p.xt[(size_t)m * p.kpad + k] = 0.f;
  if (!p.bimg) return;
  __syncthreads();
  // Terms: thread = (block bl of the tile, 32-code group gm of the tile's 64
  // codes, quarter s4): 8 MMA positions of one 32-position scale group; the
  // four quarters of a group are consecutive lanes and share its maximum.
  {
    const bool ter = p.ternary != 0;
    const int bl = tid >> 3, gm = (tid >> 2) & 1, s4 = tid & 3, b = b0 + bl;
    const bool act = b < p.nblk;
    const int64_t kk0 = (int64_t)b * p.n_b + j0;   // 64-aligned: n_b % 64 == 0
    const int64_t kb = kk0 >> 7;
    const int kl0 = (int)(kk0 & 127);
    const int g8 = (kl0 >> 3) + 4 * gm + s4;
    float v[8];
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int kl = decode_stage_k(8 * g8 + i, ter);
      v[i] = act ? tile[bl * 64 + (kl - kl0)] : 0.f;
      mx = fmaxf(mx, fabsf(v[i]));
    }
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    int ex = -125;
    if (mx > 0.f) {   // mx < 2^E, so |v 2^-(E - 2)| < 4
      int E = 0;
      frexpf(mx, &E);
      ex = E - 2;
    }
    const float inv = ldexpf(1.f, -ex);
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] *= inv;
    if (act) {
      uint8_t* img = p.bimg + (size_t)(kb >> 1) * p.NP * 128;
      const int chunk = 4 * (int)(kb & 1) + (g8 >> 2), off = 4 * (g8 & 3);
      for (int tt = 0; tt < p.T; ++tt) {
        uint32_t word = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float2 q;
          word |= e2m1x2(v[2 * i], v[2 * i + 1], &q) << (8 * i);
          v[2 * i] = (v[2 * i] - q.x) * 8.f;
          v[2 * i + 1] = (v[2 * i + 1] - q.y) * 8.f;
        }
        const int row = m * p.T + tt;
        *reinterpret_cast<uint32_t*>(img + row * 128 + ((chunk ^ (row & 7)) << 4) + off) = word;
        if (s4 == 0) p.sfbw[((size_t)kb * p.NP + row) * 4 + (g8 >> 2)] = (uint8_t)max(1, min(254, 127 + ex - 3 * tt));
      }
    }
  }
  // the K padding (the last block's second half, MMA positions 64..127 =
  // bytes 32..63 of its 64, when K_eff is an odd number of 64-code halves):
  // zero terms, unit scales
  if (jt == 0 && bt == 0 && p.kpad > p.k_eff && tid < 2 * p.T) {
    const int64_t kb = p.k_eff >> 7;
    const int tt = tid >> 1, c = 4 * (int)(kb & 1) + 2 + (tid & 1), row = m * p.T + tt;
    uint8_t* img = p.bimg + (size_t)(kb >> 1) * p.NP * 128;
    *reinterpret_cast<uint4*>(img + row * 128 + ((c ^ (row & 7)) << 4)) = make_uint4(0, 0, 0, 0);
    if ((tid & 1) == 0) {
      p.sfbw[((size_t)kb * p.NP + row) * 4 + 2] = 127;
      p.sfbw[((size_t)kb * p.NP + row) * 4 + 3] = 127;
    }
  }
}

}  // namespace

cudaError_t launch_prep(const sdq_plan_s* pl, const uint16_t* x, int M, void* ws, cudaStream_t st, float* y_zero) {
  const Geometry& g = pl->geo;
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  const int vec = (g.block % 32 == 0) && ((reinterpret_cast<uintptr_t>(x) & 15u) == 0);
  if (M <= kMaxDecodeM) {
    const DecodeConfig& dc = decode_config(pl, M);
    DecPrepParams p;
    p.x = x; p.g_hi = pl->d_g_hi; p.g_lo = pl->d_g_lo;
    p.xt = reinterpret_cast<float*>(base + L.xt);
    p.bimg = decode_image(pl) ? base + L.bimg : nullptr;
    p.sfbw = base + L.sfbw;
    p.T = dc.T; p.NP = dc.NP;
    p.y_zero = y_zero;
    p.y_count = (int64_t)M * g.n_out;
    p.ternary = g.bits == 2;
    p.M = M; p.K = g.k_in; p.B = g.block; p.n_b = g.n_b; p.nblk = g.nblk;
    p.kc = std::max(16, std::min(g.block, 256));
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
  bool used = false;
  cudaError_t et = launch_prep_tc(pl, x, M, ws, st, &used);
  if (et != cudaSuccess || used) return et;
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
