// K4 (+K6): decode contraction for batch M <= 64.
//
//   y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]
//
// (SDQ-LLM section 3.5 with eq. (12): the codes multiply the upsampled,
// Hadamard-rotated activations; every product is a signed copy of x_tilde,
// i.e. an add or a subtract.)
//
// The tiled code layout is built so that one shift and one mask of a packed
// word is a bf16 A-operand register pair of a 16x8x16 warp MMA: each half
// +-2.0 or 0, exact.  (The layout also yields fp8 registers with a wider
// mask, but sm_103 runs warp-level fp8 MMAs through conversions; bf16 is
// the native warp MMA.)  The activations enter as the B operand, written by
// the fragment kernel as bf16 hi + lo terms (hi only for M > 16); each
// (batch, term) pair is one of the 8 MMA columns.  The fp32 accumulators
// therefore hold the add/subtract sums of the codes against each term; the
// epilogue adds the terms and applies alpha / 2.
//
// Memory path: every warp streams its own sequence of 512-byte code tiles
// (16 rows x 128 / 256 codes) through a private ring of shared-memory
// slots filled with cp.async (16 bytes per lane, one commit group per tile),
// so each SM keeps ~64 KB of loads in flight without holding them in
// registers.  The CTA's slice of B-fragments arrives by one 1-D TMA bulk
// copy.  The first code tiles are requested before the grid waits on the
// fragment kernel (programmatic dependent launch), overlapping the
// activation preparation.
//
// Work split: grid (R row ranges) x (S k-slices); each warp owns whole row
// groups of its CTA's range (no CTA barrier in the stream).  With S > 1,
// per-slice partials go to the workspace and the last CTA of each row range
// (atomic ticket) sums them in slice order, so the result does not depend on
// CTA scheduling.
#include "common.cuh"

namespace sdq {

namespace {

// Occupancy and cp.async ring depth (512-byte tiles per warp) by column tiles.
__host__ __device__ constexpr int ctas_per_sm(int NT) { return NT == 1 ? 3 : (NT <= 4 ? 2 : 1); }
__host__ __device__ constexpr int ring_depth(int NT) { return NT == 1 ? 6 : (NT <= 4 ? 8 : 4); }

struct DecodeParams {
  const uint32_t* codes;
  const float* alpha;
  const uint4* frag;
  const float* scale;
  float* y;
  float* part;
  uint32_t* cnt;
  uint32_t* err;
  int M, T, n_out, ng, n_chunks;
  int S, cps, rgc, WK, WR;
};

// One tile (4 words per lane) against the bf16 B-fragments of its chunk.
// Ternary word w: (w << 2j) & 0xC000C000 is a bf16 pair, each half +-2.0 or 0
// (sign = field bit 1, exponent MSB = field bit 0).  Registers j = 0..3 form
// the A operand of one 16x8x16 MMA, j = 4..7 of a second one; the k order
// they imply is matched by the B-fragment order the fragment kernel writes.
// Binary word: ((~w << j) & 0x80008000) | 0x40004000, j = 0..15, four MMAs.
template <int QT, int NT, int QA>
__device__ __forceinline__ void mma_tile(float (&acc)[QA][NT][4], const uint32_t (&wq)[4],
                                         const uint4* bf, int lanes, bool active) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t w = wq[q];
    if (QT == 2) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t a[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) a[j] = (w << (2 * (4 * h + j))) & 0xC000C000u;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          const uint4 b = active ? bf[(q * NT + n) * lanes] : make_uint4(0, 0, 0, 0);
          mma_bf16_16816(acc[(2 * q + h) % QA][n], a, h ? b.z : b.x, h ? b.w : b.y);
        }
      }
    } else {
      const uint32_t nw = ~w;
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        uint32_t a[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) a[j] = ((nw << (4 * h + j)) & 0x80008000u) | 0x40004000u;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          // h = 0, 1: odd fields (k-steps 2q, 2q + 1); h = 2, 3: even fields
          const uint4 b = active ? bf[((2 * q + (h & 1)) * NT + n) * lanes] : make_uint4(0, 0, 0, 0);
          mma_bf16_16816(acc[(4 * q + h) % QA][n], a, (h >> 1) ? b.z : b.x, (h >> 1) ? b.w : b.y);
        }
      }
    }
  }
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

template <int QT, int NT>
__global__ void __launch_bounds__(256, ctas_per_sm(NT)) decode_kernel(DecodeParams p) {
  constexpr int KS = QT == 2 ? 4 : 8;                  // 32-code k-steps per chunk
  constexpr int QA = NT == 1 ? 4 : (NT == 2 ? 2 : 1);  // independent accumulator sets
  constexpr int D = ring_depth(NT);                    // ring slots per warp
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t frag_bar;
  __shared__ float scale_s[kMaxDecodeM];
  __shared__ int last_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = blockIdx.y, r = blockIdx.x;
  const int c0 = s * p.cps, c1 = min(p.n_chunks, c0 + p.cps);
  const int rg0 = r * p.rgc, rg1 = min(p.ng, rg0 + p.rgc);
  const int nc = c1 - c0;                                  // tiles per row group
  uint8_t* ring = smem + (size_t)warp * D * 512;          // [8 warps][D][512 B]
  uint4* bfrag = reinterpret_cast<uint4*>(smem + 8 * D * 512);
  // With one column tile only the lanes of the used columns carry fragments.
  const int flanes = NT == 1 ? 4 * p.M * p.T : 32;
  float* wb = reinterpret_cast<float*>(smem + 8 * D * 512 + (size_t)p.cps * KS * NT * flanes * 16) +
              (size_t)warp * 16 * 8 * NT;

  if (tid == 0) {
    mbar_init(&frag_bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  pdl_launch_dependents();

  // The warp's tiles: row groups rg0 + warp, rg0 + warp + 8, ...; all nc
  // chunks of the slice for each.  Each lane copies 16 of a tile's 512 bytes
  // (cp.async, one commit group per tile).  Codes do not depend on the
  // preceding kernels, so the first D - 1 tiles are requested before the
  // grid waits.
  const int n_rg_w = rg1 - rg0 - warp > 0 ? (rg1 - rg0 - warp + 7) / 8 : 0;
  const int total = n_rg_w * nc;
  const uint8_t* src = reinterpret_cast<const uint8_t*>(
      p.codes + ((size_t)(rg0 + warp) * p.n_chunks + c0) * 128) + 16 * lane;
  const size_t rg_jump = (size_t)8 * p.n_chunks * 512 - (size_t)nc * 512;
  uint8_t* dst = ring + 16 * lane;
  uint8_t* const ring_end = ring + D * 512;
  int ld_ci = 0, ld_t = 0;                                 // next tile to request
  auto request = [&]() {
    if (ld_t < total) {
      cp_async16(dst, src);
      src += 512;
      if (++ld_ci == nc) { ld_ci = 0; src += rg_jump; }
    }
    ++ld_t;
    dst += 512;
    if (dst == ring_end + 16 * lane) dst = ring + 16 * lane;
    cp_async_commit();
  };
#pragma unroll 1
  for (int d = 0; d < D - 1; ++d) request();

  // bf16 B-fragments (written by the fragment kernel) by one bulk copy.
  pdl_wait();
  const uint32_t frag_bytes = (uint32_t)(nc * KS * NT * flanes * 16);
  if (tid == 0) {
    mbar_expect_tx(&frag_bar, frag_bytes);
    bulk_g2s(bfrag, p.frag + (size_t)c0 * KS * NT * flanes, frag_bytes, &frag_bar);
  }
  if (tid < p.M) scale_s[tid] = p.scale[tid];
  const bool ok = mbar_wait(&frag_bar, 0);
  __syncthreads();
  if (!ok && tid == 0) atomicExch(p.err, 1u);

  const int g = lane >> 2, t4 = lane & 3;
  const int stride_part = p.ng * 16;
  float acc[QA][NT][4];
#pragma unroll
  for (int a = 0; a < QA; ++a)
#pragma unroll
    for (int n = 0; n < NT; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[a][n][e] = 0.f;
  int ci = 0, it = 0;
  const bool active = lane < flanes;
  const uint32_t* rd = reinterpret_cast<const uint32_t*>(ring) + lane;
  const uint32_t* const rd_end = reinterpret_cast<const uint32_t*>(ring_end) + lane;
  const uint4* bfl = bfrag + (active ? lane : 0);
#pragma unroll 1
  for (int t = 0; t < total; ++t) {
    __syncwarp();        // every lane has consumed the slot refilled next
    request();           // tile t + D - 1 into slot (t - 1) % D
    cp_async_wait<D - 1>();
    __syncwarp();        // the other lanes' copies of tile t are visible
    const uint32_t wq[4] = {rd[0], rd[32], rd[64], rd[96]};
    rd += 128;
    if (rd == rd_end) rd = reinterpret_cast<const uint32_t*>(ring) + lane;
    mma_tile<QT, NT, QA>(acc, wq, bfl + (size_t)ci * KS * NT * flanes, flanes, active);
    if (++ci == nc) {
      // Row group done: fold, stage in the warp's smem slot, combine the
      // terms of every batch row, write y (or the slice partial).
#pragma unroll
      for (int n = 0; n < NT; ++n) {
        float v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          v[e] = acc[0][n][e];
#pragma unroll
          for (int a = 1; a < QA; ++a) v[e] += acc[a][n][e];
#pragma unroll
          for (int a = 0; a < QA; ++a) acc[a][n][e] = 0.f;
        }
        const int col = n * 8 + 2 * t4;
        wb[g * 8 * NT + col] = v[0];
        wb[g * 8 * NT + col + 1] = v[1];
        wb[(g + 8) * 8 * NT + col] = v[2];
        wb[(g + 8) * 8 * NT + col + 1] = v[3];
      }
      __syncwarp();
      const int rg = rg0 + warp + 8 * it;
      for (int idx = lane; idx < 16 * p.M; idx += 32) {
        const int m = idx % p.M, row16 = idx / p.M;
        const int row = rg * 16 + row16;
        if (row < p.n_out) {
          float tot = 0.f;
          for (int term = 0; term < p.T; ++term) tot += wb[row16 * 8 * NT + m * p.T + term];
          const float val = tot / (2.f * scale_s[m]);
          if (p.S == 1)
            p.y[(size_t)m * p.n_out + row] = val * __ldg(p.alpha + row);
          else
            p.part[((size_t)s * p.M + m) * stride_part + row] = val;
        }
      }
      __syncwarp();
      ci = 0;
      ++it;
    }
  }
  cp_async_wait<0>();

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
  return launch_pdl(k, dim3(dc.R, dc.S), dim3(256), dc.smem, st, p);
}

int round_nt(int nt) { return nt <= 1 ? 1 : nt <= 2 ? 2 : nt <= 4 ? 4 : nt <= 8 ? 8 : 16; }

}  // namespace

DecodeConfig decode_config_search(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  DecodeConfig dc{};
  dc.M = M;
  dc.T = decode_terms(M);
  dc.NT = round_nt(decode_ntiles(M));
  dc.P = prep_partials(pl, M);
  dc.WK = 1;
  dc.WR = 8;
  const int KS = g.kc / 32;
  const int flanes = dc.NT == 1 ? 4 * M * dc.T : 32;
  const size_t frag_per_chunk = (size_t)KS * dc.NT * flanes * 16;
  const int cpsm = ctas_per_sm(dc.NT);
  const size_t fixed = (size_t)8 * ring_depth(dc.NT) * 512 + (size_t)8 * 16 * 8 * dc.NT * 4 + 1024;
  const size_t budget = (size_t)(cpsm == 3 ? 72 : cpsm == 2 ? 110 : 220) * 1024;
  int max_cps = (int)((budget - fixed) / frag_per_chunk);
  if (max_cps < 1) max_cps = 1;
  const int slots = pl->sm_count * cpsm;
  double best = 1e30;
  for (int S = 1; S <= g.n_chunks && S <= 64; ++S) {
    const int cps = (g.n_chunks + S - 1) / S;
    if (cps > max_cps) continue;
    if ((g.n_chunks + cps - 1) / cps != S) continue;
    // Row ranges near whole waves of CTAs, and one range per 8 groups.
    int cand[32], nc = 0;
    for (int w = 1; w <= 4; ++w) {
      const int base = (w * slots) / S;
      for (int dR = -2; dR <= 2; ++dR) cand[nc++] = base + dR;
    }
    cand[nc++] = (g.ng + 7) / 8;
    for (int ci = 0; ci < nc; ++ci) {
      const int Rr = cand[ci];
      if (Rr < 1 || Rr > g.ng) continue;
      const int rgc = (g.ng + Rr - 1) / Rr;
      const int R = (g.ng + rgc - 1) / rgc;
      const int waves = (S * R + slots - 1) / slots;
      // per-warp cost in tiles (+ an epilogue term per row group, + prologue)
      const double rg_w = (double)((rgc + 7) / 8);
      const double per = rg_w * (cps + 1.0) + (double)cps * KS * dc.NT / 512.0 + 2.0;
      const double tcost = waves * per + (S > 1 ? 0.01 * S * M : 0.0);
      if (tcost < best - 1e-9) {
        best = tcost;
        dc.S = S; dc.R = R; dc.cps = cps; dc.rgc = rgc;
      }
    }
  }
  dc.smem = (size_t)8 * ring_depth(dc.NT) * 512 + (size_t)dc.cps * frag_per_chunk +
            (size_t)8 * 16 * 8 * dc.NT * 4;
  return dc;
}

cudaError_t launch_decode(const sdq_plan_s* pl, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st) {
  const Geometry& g = pl->geo;
  const DecodeConfig& dc = decode_config(pl, M);
  const WsLayout L = workspace_layout(pl, M);
  uint8_t* base = static_cast<uint8_t*>(ws);
  DecodeParams p;
  p.codes = codes; p.alpha = alpha;
  p.frag = reinterpret_cast<const uint4*>(base + L.frag);
  p.scale = reinterpret_cast<const float*>(base + L.scale);
  p.part = reinterpret_cast<float*>(base + L.part);
  p.cnt = reinterpret_cast<uint32_t*>(base + L.cnt);
  p.err = reinterpret_cast<uint32_t*>(base + L.err);
  p.y = y;
  p.M = M; p.T = dc.T; p.n_out = g.n_out; p.ng = g.ng; p.n_chunks = g.n_chunks;
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
