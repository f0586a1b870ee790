// K4 (+K6): decode contraction for batch M <= 64.
//
//   y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]
//
// (SDQ-LLM section 3.5 with eq. (12): the codes multiply the upsampled,
// Hadamard-rotated activations; every product is a signed copy of x_tilde,
// i.e. an add or a subtract.)
//
// The tiled code layout is built so that one shift and one mask of a packed
// word is an fp8 (e4m3) A-operand register of a 16x8x32 warp MMA: each byte
// +-2.0 or 0, exact.  The activations enter as the B operand, written as a
// T-term fp8 expansion  x_tilde * s = t0 + t1/16 + t2/256  (T = 3 for M <= 2,
// else 2) with a power-of-two scale s per batch row; each (batch, term) pair
// is one of the 8 MMA columns.  The fp32 accumulators therefore carry the
// add/subtract sums of the codes against each term; the epilogue recombines
// the terms and applies alpha.
//
// Work split: grid (R row ranges) x (S k-slices).  A CTA stages the fp8
// B-fragments of its k-slice in shared memory once, then its 8 warps stream
// the tiled codes of their row groups straight from HBM (coalesced 128-byte
// warp loads, one tile of 16 rows x 128/256 codes at a time, prefetched one
// tile ahead).  WK warps split the k-slice of one row group and reduce
// through shared memory.  With S > 1, per-slice partials go to the workspace
// and the last CTA of each row range (atomic ticket) sums them in slice
// order, so the result does not depend on CTA scheduling.
#include "common.cuh"

namespace sdq {

namespace {

struct DecodeParams {
  const uint32_t* codes;
  const float* alpha;
  const float* xt;
  const float* pmax;
  float* y;
  float* part;
  uint32_t* cnt;
  int M, T, n_out, ng, n_chunks, P;
  int64_t kpad;
  int S, cps, rgc, WK, WR;
};

__device__ __forceinline__ uint32_t fp8_term(float v, int term) {
  uint32_t b = f32_to_e4m3(v);
  if (term == 0) return b;
  float r = (v - e4m3_to_f32(b)) * 16.f;
  b = f32_to_e4m3(r);
  if (term == 1) return b;
  r = (r - e4m3_to_f32(b)) * 16.f;
  return f32_to_e4m3(r);
}

template <int QT, int NT>
__global__ void __launch_bounds__(256) decode_kernel(DecodeParams p) {
  constexpr int KS = QT == 2 ? 4 : 8;        // 32-code k-steps per chunk
  constexpr int QA = NT == 1 ? 4 : (NT == 2 ? 2 : 1);  // independent accumulator sets
  extern __shared__ __align__(16) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = blockIdx.y, r = blockIdx.x;
  const int c0 = s * p.cps, c1 = min(p.n_chunks, c0 + p.cps);
  const int rg0 = r * p.rgc, rg1 = min(p.ng, rg0 + p.rgc);
  const int nks = (c1 - c0) * KS;

  uint2* bfrag = reinterpret_cast<uint2*>(smem);
  float* wred = reinterpret_cast<float*>(smem + (size_t)p.cps * KS * NT * 32 * sizeof(uint2));
  float* scale_s = wred + 8 * 16 * 8 * NT;
  __shared__ int last_flag;

  // Power-of-two scale per batch row: max |x_tilde| * s in [128, 256).
  if (tid < p.M) {
    float amax = 0.f;
    for (int i = 0; i < p.P; ++i) amax = fmaxf(amax, p.pmax[(size_t)tid * p.P + i]);
    float sc = 1.f;
    if (amax > 0.f) {
      int e;
      frexpf(amax, &e);
      sc = ldexpf(1.f, 8 - e);
    }
    scale_s[tid] = sc;
  }
  __syncthreads();
  // fp8 B-fragments of the slice: lane (g, t) of k-step ks holds, for column
  // n = 8 nt + g, bytes k = 32 ks + 4t + {0..3} (b0) and + 16 (b1).
  const int cols = p.M * p.T;
  for (int idx = tid; idx < nks * NT * 32; idx += 256) {
    const int ln = idx & 31, nt = (idx >> 5) % NT, ks = idx / (32 * NT);
    const int g = ln >> 2, t = ln & 3, n = nt * 8 + g;
    uint32_t b0 = 0, b1 = 0;
    if (n < cols) {
      const int m = n / p.T, term = n - m * p.T;
      const float sc = scale_s[m];
      const float* xr = p.xt + (size_t)m * p.kpad + (size_t)(c0 * KS + ks) * 32 + 4 * t;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        b0 |= fp8_term(xr[i] * sc, term) << (8 * i);
        b1 |= fp8_term(xr[16 + i] * sc, term) << (8 * i);
      }
    }
    bfrag[idx] = make_uint2(b0, b1);
  }
  __syncthreads();

  const int WK = p.WK, WR = p.WR;
  const int wr = warp / WK, wk = warp - wr * WK;
  const int g = lane >> 2, t = lane & 3;
  const int stride_part = p.ng * 16;

  for (int rgb = rg0; rgb < rg1; rgb += WR) {
    const int rg = rgb + wr;
    float acc[QA][NT][4];
#pragma unroll
    for (int a = 0; a < QA; ++a)
#pragma unroll
      for (int n = 0; n < NT; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[a][n][e] = 0.f;
    if (rg < rg1) {
      const uint32_t* tb = p.codes + (size_t)rg * p.n_chunks * 128 + lane;
      int c = c0 + wk;
      uint32_t wcur[4] = {0, 0, 0, 0}, wnxt[4] = {0, 0, 0, 0};
      if (c < c1) {
#pragma unroll
        for (int q = 0; q < 4; ++q) wcur[q] = __ldcs(tb + (size_t)c * 128 + 32 * q);
      }
      for (; c < c1; c += WK) {
        const int cn = c + WK;
        if (cn < c1) {
#pragma unroll
          for (int q = 0; q < 4; ++q) wnxt[q] = __ldcs(tb + (size_t)cn * 128 + 32 * q);
        }
        const uint2* bf = bfrag + (size_t)(c - c0) * KS * NT * 32 + lane;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint32_t w = wcur[q];
          if (QT == 2) {
            uint32_t a[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) a[j] = (w << (2 * j)) & 0xC0C0C0C0u;
#pragma unroll
            for (int n = 0; n < NT; ++n) {
              const uint2 b = bf[(q * NT + n) * 32];
              mma_e4m3_16832(acc[q % QA][n], a, b.x, b.y);
            }
          } else {
            const uint32_t nw = ~w;
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              uint32_t a[4];
#pragma unroll
              for (int j = 0; j < 4; ++j) a[j] = ((nw << (4 * u + j)) & 0x80808080u) | 0x40404040u;
#pragma unroll
              for (int n = 0; n < NT; ++n) {
                const uint2 b = bf[((2 * q + u) * NT + n) * 32];
                mma_e4m3_16832(acc[(2 * q + u) % QA][n], a, b.x, b.y);
              }
            }
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) wcur[q] = wnxt[q];
      }
    }
    // Fold accumulator sets and stage per-warp sums: wred[warp][row][col].
    float* wb = wred + (size_t)warp * 16 * 8 * NT;
#pragma unroll
    for (int n = 0; n < NT; ++n) {
      float v[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[e] = acc[0][n][e];
#pragma unroll
        for (int a = 1; a < QA; ++a) v[e] += acc[a][n][e];
      }
      const int col = n * 8 + 2 * t;
      wb[g * 8 * NT + col] = v[0];
      wb[g * 8 * NT + col + 1] = v[1];
      wb[(g + 8) * 8 * NT + col] = v[2];
      wb[(g + 8) * 8 * NT + col + 1] = v[3];
    }
    __syncthreads();
    // Combine the WK k-split warps and the fp8 terms of every batch row.
    for (int idx = tid; idx < WR * 16 * p.M; idx += 256) {
      const int m = idx % p.M, rr = idx / p.M, wrr = rr >> 4, row16 = rr & 15;
      const int row = (rgb + wrr) * 16 + row16;
      if (rgb + wrr < rg1 && row < p.n_out) {
        float tot = 0.f, wgt = 1.f;
        for (int term = 0; term < p.T; ++term) {
          const int col = m * p.T + term;
          float sum = 0.f;
          for (int k = 0; k < WK; ++k)
            sum += wred[((size_t)(wrr * WK + k) * 16 + row16) * 8 * NT + col];
          tot += sum * wgt;
          wgt *= 0.0625f;
        }
        const float val = tot / (2.f * scale_s[m]);
        if (p.S == 1)
          p.y[(size_t)m * p.n_out + row] = val * __ldg(p.alpha + row);
        else
          p.part[((size_t)s * p.M + m) * stride_part + row] = val;
      }
    }
    __syncthreads();
  }

  if (p.S > 1) {
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const uint32_t prev = atomicAdd(p.cnt + r, 1u);
      last_flag = prev == (uint32_t)(p.S - 1);
    }
    __syncthreads();
    if (last_flag) {
      __threadfence();
      const int row_lo = rg0 * 16, row_hi = min(p.n_out, rg1 * 16);
      for (int idx = tid; idx < (row_hi - row_lo) * p.M; idx += 256) {
        const int m = idx / (row_hi - row_lo), row = row_lo + idx % (row_hi - row_lo);
        float v = 0.f;
        for (int ss = 0; ss < p.S; ++ss) v += __ldcg(p.part + ((size_t)ss * p.M + m) * stride_part + row);
        p.y[(size_t)m * p.n_out + row] = v * __ldg(p.alpha + row);
      }
      if (tid == 0) p.cnt[r] = 0u;
    }
  }
}

template <int QT, int NT>
cudaError_t launch_t(const DecodeConfig& dc, const DecodeParams& p, cudaStream_t st) {
  auto k = decode_kernel<QT, NT>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dc.smem);
  if (e != cudaSuccess) return e;
  dim3 grid(dc.R, dc.S);
  k<<<grid, 256, dc.smem, st>>>(p);
  return cudaGetLastError();
}

int round_nt(int nt) { return nt <= 1 ? 1 : nt <= 2 ? 2 : nt <= 4 ? 4 : nt <= 8 ? 8 : 16; }

}  // namespace

DecodeConfig decode_config_search(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  DecodeConfig dc{};
  dc.M = M;
  dc.T = decode_terms(M);
  dc.NT = round_nt(decode_ntiles(M));
  const int KS = g.kc / 32;
  const int JT = (g.n_b + 63) / 64, BT = (g.nblk + 63) / 64;
  dc.P = JT * BT;
  const size_t frag_per_chunk = (size_t)KS * dc.NT * 32 * 8;
  const size_t fixed = (size_t)8 * 16 * 8 * dc.NT * 4 + 64 * 4 + 64;
  const int ctas_per_sm = dc.NT <= 2 ? 2 : 1;
  const size_t budget = (ctas_per_sm == 2 ? 110 : 220) * 1024;
  int max_cps = (int)((budget - fixed) / frag_per_chunk);
  if (max_cps < 1) max_cps = 1;
  const int slots = pl->sm_count * ctas_per_sm;
  double best = 1e30;
  for (int S = 1; S <= g.n_chunks && S <= 64; ++S) {
    const int cps = (g.n_chunks + S - 1) / S;
    if (cps > max_cps) continue;
    const int S_eff = (g.n_chunks + cps - 1) / cps;
    if (S_eff != S) continue;
    for (int WK = 1; WK <= 8; WK *= 2) {
      if (WK > cps) break;
      const int WR = 8 / WK;
      // Row ranges: values near whole waves of CTAs, and one range per group.
      int cand[32], nc = 0;
      for (int w = 1; w <= 4; ++w) {
        const int base = (w * slots) / S;
        for (int dR = -2; dR <= 2; ++dR) cand[nc++] = base + dR;
      }
      cand[nc++] = g.ng;
      for (int ci = 0; ci < nc; ++ci) {
        const int Rr = cand[ci];
        if (Rr < 1 || Rr > g.ng) continue;
        const int rgc = (g.ng + Rr - 1) / Rr;
        const int R = (g.ng + rgc - 1) / rgc;
        const int ctas = S * R;
        const int waves = (ctas + slots - 1) / slots;
        // per-CTA cost in tile loads per warp, plus sync and prologue terms
        const double iters = (double)((rgc + WR - 1) / WR);
        const double per = iters * (double)((cps + WK - 1) / WK) + iters * 1.5 +
                           (double)cps * KS * dc.NT / 64.0 + 4.0;
        const double tcost = waves * per + (S > 1 ? 0.02 * S * M : 0.0);
        if (tcost < best - 1e-9) {
          best = tcost;
          dc.S = S; dc.R = R; dc.WK = WK; dc.WR = WR; dc.cps = cps; dc.rgc = rgc;
        }
      }
    }
  }
  dc.smem = (size_t)dc.cps * frag_per_chunk + (size_t)8 * 16 * 8 * dc.NT * 4 + 64 * 4;
  return dc;
}

cudaError_t launch_decode(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  const DecodeConfig dc = decode_config(pl, M);
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  DecodeParams p;
  p.codes = codes; p.alpha = alpha;
  p.xt = reinterpret_cast<const float*>(base + L.xt);
  p.pmax = reinterpret_cast<const float*>(base + L.pmax);
  p.part = reinterpret_cast<float*>(base + L.part);
  p.cnt = reinterpret_cast<uint32_t*>(base + L.cnt);
  p.y = y;
  p.M = M; p.T = dc.T; p.n_out = g.n_out; p.ng = g.ng; p.n_chunks = g.n_chunks; p.P = dc.P;
  p.kpad = g.k_eff_pad;
  p.S = dc.S; p.cps = dc.cps; p.rgc = dc.rgc; p.WK = dc.WK; p.WR = dc.WR;
  const bool tern = pl->desc.quantizer == SDQ_TERNARY;
  switch (dc.NT) {
    case 1: return tern ? launch_t<2, 1>(dc, p, st) : launch_t<1, 1>(dc, p, st);
    case 2: return tern ? launch_t<2, 2>(dc, p, st) : launch_t<1, 2>(dc, p, st);
    case 4: return tern ? launch_t<2, 4>(dc, p, st) : launch_t<1, 4>(dc, p, st);
    case 8: return tern ? launch_t<2, 8>(dc, p, st) : launch_t<1, 8>(dc, p, st);
    default: return tern ? launch_t<2, 16>(dc, p, st) : launch_t<1, 16>(dc, p, st);
  }
}

}  // namespace sdq
