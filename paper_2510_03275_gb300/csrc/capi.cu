// C ABI of libsdq (declarations and contracts in include/sdq.h).
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <numeric>
#include <vector>

#include "common.cuh"

namespace sdq {

namespace {

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

uint16_t host_bf16(double v) {
  float f = (float)v;
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}
double host_bf16_value(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

int cuda_status(cudaError_t e) { return e == cudaSuccess ? SDQ_OK : SDQ_ERR_CUDA; }

// The polyphase table of D^T (layout: poly_stride in sdq_internal.h) from
// D^T itself (n_b x B, fp64).  Sets p, q (n_b / B = p / q in lowest terms)
// always; fills `poly` and returns SDQ_OK when the decode kernel can use it:
// B a multiple of 16 up to kMaxPolyBlock, n_b a multiple of 8, the entries
// within kMaxPolyBytes, and D^T polyphase to 1e-12 of its largest entry.
int build_poly_table(const Geometry& g, const sdq_layer_desc* desc, const int8_t* had_signs,
                     const std::vector<double>& dt, std::vector<uint32_t>* poly, int* p_out, int* q_out) {
  const int B = g.block, pp = g.n_b / std::gcd(g.n_b, g.block), pq = g.block / std::gcd(g.n_b, g.block);
  *p_out = pp;
  *q_out = pq;
  const size_t poly_bytes = (size_t)pp * poly_stride(B) * 8;
  if (B % 16 != 0 || g.n_b % 8 != 0 || B > kMaxPolyBlock || poly_bytes > (size_t)kMaxPolyBytes)
    return SDQ_ERR_UNSUPPORTED;
  const size_t tab = (size_t)g.n_b * B;
  double mx = 0.0, dev = 0.0;
  for (size_t i = 0; i < tab; ++i) mx = std::max(mx, std::fabs(dt[i]));
  for (int j = 0; j < g.n_b; ++j)
    for (int i = 0; i < B; ++i) {
      const int src = (int)(((int64_t)i - (int64_t)pq * (j / pp)) % B + B) % B;
      dev = std::max(dev, std::fabs(dt[(size_t)j * B + i] - dt[(size_t)(j % pp) * B + src]));
    }
  if (dev > 1e-12 * mx) return SDQ_ERR_UNSUPPORTED;
  poly->assign(poly_bytes / 4 + B, 0u);
  for (int r = 0; r < pp; ++r)
    for (int d = 0; d < 2 * B; ++d) {
      uint32_t hi = 0, lo = 0;
      for (int h = 0; h < 2; ++h) {   // taps d and d + 1 (mod B): low and high halves
        double v = dt[(size_t)r * B + (d + h) % B];
        if (std::fabs(v) < 0x1p-46) v = 0.0;   // fp64 noise on exact zeros
        const uint16_t vh = host_bf16(v), vl = host_bf16(v - host_bf16_value(vh));
        hi |= (uint32_t)vh << (16 * h);
        lo |= (uint32_t)vl << (16 * h);
      }
      const size_t e = (size_t)r * poly_stride(B) + d;
      (*poly)[2 * e] = hi;
      (*poly)[2 * e + 1] = lo;
    }
  const bool had = desc->hadamard != 0;
  for (int k = 0; k < B; ++k) {
    const float sk = had ? (float)((had_signs ? (double)had_signs[k] : 1.0) / std::sqrt((double)B)) : 1.0f;
    std::memcpy(&(*poly)[poly_bytes / 4 + k], &sk, 4);
  }
  return SDQ_OK;
}

}  // namespace

uint64_t next_call_number() {
  static std::atomic<uint64_t> calls{0};
  return ++calls;
}

WsLayout workspace_layout(const sdq_plan_s* pl, int M) {
  const Geometry& g = pl->geo;
  WsLayout L{};
  size_t off = 0;
  L.xt = off;
  if (M <= kMaxDecodeM) {
    const DecodeConfig& dc = pl->dcfg[M];
    off = align_up(off + sizeof(float) * (size_t)M * g.k_eff_pad, 256);
    L.bimg = off;                                  // e4m3 B operand image, K/128 x NP x 128 bytes
    off = align_up(off + (size_t)(g.k_eff_pad / 128) * dc.NP * 128, 256);
    L.sexp = off;                                  // per-batch-row scale exponents
    off = align_up(off + sizeof(int32_t) * kMaxDecodeM, 256);
    L.part = off;
    off = align_up(off + (dc.S > 1 ? sizeof(float) * (size_t)dc.S * M * g.ntiles * kTileRows : 0), 256);
    L.cnt = off;                                   // one 64-bit ticket per row tile
    off = align_up(off + sizeof(uint64_t) * (size_t)g.ntiles, 256);
    L.err = off;                                   // call record
    off = align_up(off + 2 * sizeof(uint64_t), 256);
  } else {
    off = align_up(off + sizeof(uint16_t) * (size_t)M * g.k_eff_pad, 256);
    L.bimg = L.sexp = L.part = L.cnt = L.err = off;   // call record only
    off = align_up(off + 2 * sizeof(uint64_t), 256);
  }
  L.total = off;
  return L;
}

}  // namespace sdq

using namespace sdq;

extern "C" int sdq_plan_create(const sdq_layer_desc* desc, const int8_t* had_signs, sdq_plan* out) {
  if (!desc || !out) return SDQ_ERR_INVALID_ARG;
  *out = nullptr;
  Geometry g;
  int st = validate(desc, &g);
  if (st != SDQ_OK) return st;
  int dev = 0, major = 0, minor = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDQ_ERR_CUDA;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return SDQ_ERR_CUDA;
  if (major != 10 || minor != 3) return SDQ_ERR_UNSUPPORTED;

  const size_t tab = (size_t)g.n_b * g.block;
  std::vector<float> a_enc(tab), gm(tab), at(tab);
  std::vector<double> dt(tab);
  st = build_tables(desc, had_signs, a_enc.data(), gm.data(), dt.data());
  if (st != SDQ_OK) return st;
  for (int j = 0; j < g.n_b; ++j)
    for (int k = 0; k < g.block; ++k) at[(size_t)k * g.n_b + j] = a_enc[(size_t)j * g.block + k];
  // max_j sum_k |G[j][k]|, with a margin for the bf16 hi + lo split of G
  double gnorm = 0.0;
  for (int j = 0; j < g.n_b; ++j) {
    double sr = 0.0;
    for (int k = 0; k < g.block; ++k) sr += std::fabs((double)gm[(size_t)j * g.block + k]);
    gnorm = std::max(gnorm, sr);
  }
  std::vector<uint16_t> ghi(tab), glo(tab);
  for (size_t i = 0; i < tab; ++i) {
    ghi[i] = host_bf16(gm[i]);
    glo[i] = host_bf16((double)gm[i] - host_bf16_value(ghi[i]));
  }

  std::vector<uint16_t> gfrag;
  if (g.block % 16 == 0 && g.n_b % 8 == 0) {
    const int kbw = g_frag_batch(g.block), R = kbw / 4, nkb = g.block / kbw;
    gfrag.resize(2 * tab);
    for (int jt = 0; jt < g.n_b / 8; ++jt)
      for (int kb = 0; kb < nkb; ++kb)
        for (int lane = 0; lane < 32; ++lane) {
          const int j = 8 * jt + (lane >> 2), t = lane & 3;
          uint16_t* dst = gfrag.data() + (size_t)2 * R * (32 * ((size_t)jt * nkb + kb) + lane);
          const size_t src = (size_t)j * g.block + (size_t)kb * kbw + (size_t)t * R;
          for (int e = 0; e < R; ++e) {   // 32-bit words alternate hi, lo
            dst[4 * (e >> 1) + (e & 1)] = ghi[src + e];
            dst[4 * (e >> 1) + 2 + (e & 1)] = glo[src + e];
          }
        }
  }

  // Polyphase table of D^T (poly_stride) when D^T has that structure to fp64
  // rounding and the table is small (else the decode build streams G).
  std::vector<uint32_t> poly;
  int pp = 0, pq = 0;
  if (build_poly_table(g, desc, had_signs, dt, &poly, &pp, &pq) != SDQ_OK) poly.clear();
  const size_t poly_bytes = (size_t)pp * poly_stride(g.block) * 8;

  sdq_plan_s* p = new (std::nothrow) sdq_plan_s();
  if (!p) return SDQ_ERR_ALLOC;
  p->poly_p = pp;
  p->poly_q = pq;
  p->poly_bytes = (int)poly_bytes;
  p->desc = *desc;
  p->geo = g;
  p->device = dev;
  p->sm_count = sms;
  p->gnorm = (float)(gnorm * (1.0 + 1.0 / 1024));
  if (cudaMalloc(&p->d_at, sizeof(float) * tab) != cudaSuccess ||
      cudaMalloc(&p->d_g_hi, sizeof(uint16_t) * tab) != cudaSuccess ||
      cudaMalloc(&p->d_g_lo, sizeof(uint16_t) * tab) != cudaSuccess ||
      (!gfrag.empty() && cudaMalloc(&p->d_g_frag, sizeof(uint16_t) * gfrag.size()) != cudaSuccess) ||
      (!poly.empty() && cudaMalloc(&p->d_poly, sizeof(uint32_t) * poly.size()) != cudaSuccess)) {
    sdq_plan_destroy(p);
    return SDQ_ERR_ALLOC;
  }
  if (cudaMemcpy(p->d_at, at.data(), sizeof(float) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(p->d_g_hi, ghi.data(), sizeof(uint16_t) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(p->d_g_lo, glo.data(), sizeof(uint16_t) * tab, cudaMemcpyHostToDevice) != cudaSuccess ||
      (!gfrag.empty() && cudaMemcpy(p->d_g_frag, gfrag.data(), sizeof(uint16_t) * gfrag.size(),
                                    cudaMemcpyHostToDevice) != cudaSuccess) ||
      (!poly.empty() && cudaMemcpy(p->d_poly, poly.data(), sizeof(uint32_t) * poly.size(),
                                   cudaMemcpyHostToDevice) != cudaSuccess)) {
    sdq_plan_destroy(p);
    return SDQ_ERR_CUDA;
  }
  for (int M = 1; M <= kMaxDecodeM; ++M) p->dcfg[M] = decode_config_search(p, M);
  *out = p;
  return SDQ_OK;
}

extern "C" int sdq_build_poly_table(const sdq_layer_desc* desc, const int8_t* had_signs, uint32_t* table,
                                    size_t capacity_words, size_t* words_out, int32_t* p_out, int32_t* q_out) {
  if (!desc) return SDQ_ERR_INVALID_ARG;
  Geometry g;
  int st = validate(desc, &g);
  if (st != SDQ_OK) return st;
  std::vector<double> dt((size_t)g.n_b * g.block);
  st = build_tables(desc, had_signs, nullptr, nullptr, dt.data());
  if (st != SDQ_OK) return st;
  std::vector<uint32_t> poly;
  int pp = 0, pq = 0;
  st = build_poly_table(g, desc, had_signs, dt, &poly, &pp, &pq);
  if (p_out) *p_out = pp;
  if (q_out) *q_out = pq;
  if (words_out) *words_out = poly.size();
  if (st != SDQ_OK) return st;
  if (table) {
    if (capacity_words < poly.size()) return SDQ_ERR_WORKSPACE;
    std::memcpy(table, poly.data(), sizeof(uint32_t) * poly.size());
  }
  return SDQ_OK;
}

extern "C" int sdq_plan_destroy(sdq_plan p) {
  if (!p) return SDQ_ERR_INVALID_ARG;
  cudaError_t e = cudaSuccess, e2;
  if (p->d_at && (e2 = cudaFree(p->d_at)) != cudaSuccess) e = e2;
  if (p->d_g_hi && (e2 = cudaFree(p->d_g_hi)) != cudaSuccess) e = e2;
  if (p->d_g_lo && (e2 = cudaFree(p->d_g_lo)) != cudaSuccess) e = e2;
  if (p->d_g_frag && (e2 = cudaFree(p->d_g_frag)) != cudaSuccess) e = e2;
  if (p->d_poly && (e2 = cudaFree(p->d_poly)) != cudaSuccess) e = e2;
  delete p;
  return cuda_status(e);
}

extern "C" size_t sdq_workspace_bytes(sdq_plan p, int32_t M) {
  if (!p || M < 1 || M > (1 << 20)) return 0;
  return workspace_layout(p, M).total;
}

extern "C" int sdq_encode_rows(sdq_plan p, const float* W, uint32_t* codes_plain, float* alpha,
                               void* stream) {
  if (!p || !W || !codes_plain || !alpha) return SDQ_ERR_INVALID_ARG;
  if (!aligned16(W) || !aligned16(codes_plain) || !aligned16(alpha)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_encode(p, W, codes_plain, alpha, (cudaStream_t)stream));
}

extern "C" int sdq_pack(sdq_plan p, const uint32_t* plain, uint32_t* tiled, void* stream) {
  if (!p || !plain || !tiled || !aligned16(plain) || !aligned16(tiled)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_pack(p, plain, tiled, (cudaStream_t)stream));
}

extern "C" int sdq_unpack(sdq_plan p, const uint32_t* tiled, uint32_t* plain, uint32_t* bad_count,
                          void* stream) {
  if (!p || !plain || !tiled || !aligned16(plain) || !aligned16(tiled)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_unpack(p, tiled, plain, bad_count, (cudaStream_t)stream));
}

static int check_ws(sdq_plan p, int32_t M, const void* ws, size_t ws_bytes) {
  if (!p || M < 1 || M > 65535) return SDQ_ERR_INVALID_ARG;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u)) return SDQ_ERR_INVALID_ARG;
  if (ws_bytes < workspace_layout(p, M).total) return SDQ_ERR_WORKSPACE;
  return SDQ_OK;
}

extern "C" int sdq_prep_activations(sdq_plan p, const uint16_t* x, int32_t M, void* ws,
                                    size_t ws_bytes, void* stream) {
  int st = check_ws(p, M, ws, ws_bytes);
  if (st != SDQ_OK) return st;
  if (!x || !aligned16(x)) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_prep(p, x, M, ws, (cudaStream_t)stream));
}

static int contract(sdq_plan p, const uint32_t* codes_tiled, const float* alpha, int32_t M, float* y,
                    void* ws, size_t ws_bytes, void* stream, int early, const uint16_t* x_fused) {
  int st = check_ws(p, M, ws, ws_bytes);
  if (st != SDQ_OK) return st;
  if (!codes_tiled || !alpha || !y || !aligned16(codes_tiled) || !aligned16(y)) return SDQ_ERR_INVALID_ARG;
  cudaError_t e = M <= kMaxDecodeM
                      ? launch_decode(p, codes_tiled, alpha, M, y, ws, (cudaStream_t)stream, early, x_fused)
                      : launch_prefill(p, codes_tiled, alpha, M, y, ws, (cudaStream_t)stream);
  if (e == cudaErrorNotSupported) return SDQ_ERR_UNSUPPORTED;
  return cuda_status(e);
}

extern "C" int sdq_contract(sdq_plan p, const uint32_t* codes_tiled, const float* alpha, int32_t M,
                            float* y, void* ws, size_t ws_bytes, void* stream) {
  return contract(p, codes_tiled, alpha, M, y, ws, ws_bytes, stream, 0, nullptr);
}

// Small decode batches: one kernel that builds its own B operand from x.
// Otherwise the prepare kernel, then the contraction; behind its own prepare
// kernel the decode kernel may start reading the codes before the preceding
// grid finishes: that grid waited for everything before it in the stream, and
// it does not write the codes.
extern "C" int sdq_linear_forward(sdq_plan p, const uint32_t* codes_tiled, const float* alpha,
                                  const uint16_t* x, int32_t M, float* y, void* ws, size_t ws_bytes,
                                  void* stream) {
  if (p && x && M >= 1 && M <= kMaxDecodeM && decode_fusable(p, M, x))
    return contract(p, codes_tiled, alpha, M, y, ws, ws_bytes, stream, 0, x);
  int st = sdq_prep_activations(p, x, M, ws, ws_bytes, stream);
  if (st != SDQ_OK) return st;
  return contract(p, codes_tiled, alpha, M, y, ws, ws_bytes, stream, 1, nullptr);
}

extern "C" int sdq_forward_kernels(sdq_plan p, int32_t M, const uint16_t* x) {
  if (!p || !x || M < 1 || M > 65535) return 0;
  return M <= kMaxDecodeM && decode_fusable(p, M, x) ? 1 : 2;
}

extern "C" int sdq_workspace_status(sdq_plan p, int32_t M, const void* ws, void* stream) {
  if (!p || M < 1 || M > 65535 || !ws) return SDQ_ERR_INVALID_ARG;
  const WsLayout L = workspace_layout(p, M);
  uint64_t rec[2] = {0, 0};   // last failed call, last call
  cudaError_t e = cudaMemcpyAsync(rec, static_cast<const uint8_t*>(ws) + L.err, sizeof(rec),
                                  cudaMemcpyDeviceToHost, (cudaStream_t)stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return SDQ_ERR_CUDA;
  return rec[1] != 0 && rec[0] == rec[1] ? SDQ_ERR_TIMEOUT : SDQ_OK;
}

extern "C" int sdq_read_prep(sdq_plan p, int32_t M, const void* ws, float* xt_out, void* stream) {
  if (!p || M < 1 || M > kMaxDecodeM || !ws || !xt_out) return SDQ_ERR_INVALID_ARG;
  return cuda_status(launch_read_prep(p, M, ws, xt_out, (cudaStream_t)stream));
}

namespace sdq {

namespace {
__global__ void read_prep_kernel(const float* xt, float* out, int M, int64_t k_eff, int64_t kpad) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)M * k_eff) return;
  const int64_t m = i / k_eff, k = i - m * k_eff;
  out[i] = xt[m * kpad + k];
}
}  // namespace

cudaError_t launch_read_prep(const sdq_plan_s* p, int M, const void* ws, float* out, cudaStream_t st) {
  const WsLayout L = workspace_layout(p, M);
  const float* xt = reinterpret_cast<const float*>(static_cast<const uint8_t*>(ws) + L.xt);
  const int64_t n = (int64_t)M * p->geo.k_eff;
  read_prep_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(xt, out, M, p->geo.k_eff, p->geo.k_eff_pad);
  return cudaGetLastError();
}

}  // namespace sdq
