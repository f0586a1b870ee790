// GPTQ block compensation for the Sigma-Delta encoder (SDQ-LLM Algorithm 1:
// the outer loop over blocks of B columns, with the inverse Hessian H^-1 =
// (2 X X^T + lambda I)^-1 given through its upper Cholesky factor U,
// U^T U = H^-1).
//
// Blocks are encoded in order on a working copy of W.  After block b is
// encoded (encode_kernel, one block per launch), each row's block error E =
// W_F - alpha (c . G) is normalised by the factor's diagonal block, E~ =
// E U_FF^-1, and the later columns take the update W_R -= E~ U_FR: the exact
// block update of GPTQ / optimal brain surgeon (for B = 1 it is GPTQ's
// division by the diagonal), equal to E H_FR H_RR^-1.  Every product and sum
// is a rounded fp32 operation in a fixed order (ascending k, first product
// not added to a zero), so the codes are a deterministic function of W and U.
#include "encode.cuh"

namespace sdq {

namespace {

constexpr int kUpT = 128;      // rows and columns of W per CTA
constexpr int kUpK = 32;       // block columns (k) per shared-memory chunk
constexpr int kUpThreads = 256;

// W[r, c] -= sum_k E~[r, k] U[f0 + k, c] for r < n_out, c in [col0, k_in):
// 128 x 128 outputs per CTA, 8 x 8 per thread (rows 4 ty .. 4 ty + 3 and 64 +
// the same, columns likewise in tx), E~ and U staged through shared memory
// 32 k at a time.
__global__ void __launch_bounds__(kUpThreads, 2)
    gptq_update_kernel(float* __restrict__ W, const float* __restrict__ et, const float* __restrict__ U,
                       int n_out, int k_in, int B, int f0, int col0) {
  __shared__ __align__(16) float es[kUpK][kUpT];   // es[k][row] = E~[r0 + row, kc + k]
  __shared__ __align__(16) float us[kUpK][kUpT];   // us[k][col] = U[f0 + kc + k, c0 + col]
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int r0 = blockIdx.y * kUpT, c0 = col0 + blockIdx.x * kUpT;
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = -0.0f;   // -0 + p == p: the first product is taken as is
  for (int kc = 0; kc < B; kc += kUpK) {
    const int kn = min(kUpK, B - kc);
    for (int i = tid; i < kUpT * (kUpK / 4); i += kUpThreads) {
      const int row = i / (kUpK / 4), k4 = i % (kUpK / 4);
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (r0 + row < n_out && 4 * k4 < kn)
        v = __ldg(reinterpret_cast<const float4*>(et + (size_t)(r0 + row) * B + kc + 4 * k4));
      es[4 * k4 + 0][row] = v.x;
      es[4 * k4 + 1][row] = v.y;
      es[4 * k4 + 2][row] = v.z;
      es[4 * k4 + 3][row] = v.w;
    }
    for (int i = tid; i < kUpK * (kUpT / 4); i += kUpThreads) {
      const int k = i / (kUpT / 4), c4 = i % (kUpT / 4);
      const int col = c0 + 4 * c4;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (k < kn && col < k_in)
        v = __ldg(reinterpret_cast<const float4*>(U + (size_t)(f0 + kc + k) * k_in + col));
      *reinterpret_cast<float4*>(&us[k][4 * c4]) = v;
    }
    __syncthreads();
    for (int k = 0; k < kn; ++k) {
      float a[8], b[8];
      *reinterpret_cast<float4*>(&a[0]) = *reinterpret_cast<const float4*>(&es[k][4 * ty]);
      *reinterpret_cast<float4*>(&a[4]) = *reinterpret_cast<const float4*>(&es[k][64 + 4 * ty]);
      *reinterpret_cast<float4*>(&b[0]) = *reinterpret_cast<const float4*>(&us[k][4 * tx]);
      *reinterpret_cast<float4*>(&b[4]) = *reinterpret_cast<const float4*>(&us[k][64 + 4 * tx]);
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = __fadd_rn(acc[i][j], __fmul_rn(a[i], b[j]));
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int row = r0 + (i < 4 ? 4 * ty + i : 64 + 4 * ty + i - 4);
    if (row >= n_out) continue;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int col = c0 + 64 * h + 4 * tx;   // k_in and col are multiples of 4
      if (col >= k_in) continue;
      float4* wp = reinterpret_cast<float4*>(W + (size_t)row * k_in + col);
      float4 w = *wp;
      w.x = __fsub_rn(w.x, acc[i][4 * h + 0]);
      w.y = __fsub_rn(w.y, acc[i][4 * h + 1]);
      w.z = __fsub_rn(w.z, acc[i][4 * h + 2]);
      w.w = __fsub_rn(w.w, acc[i][4 * h + 3]);
      *wp = w;
    }
  }
}

inline size_t align256(size_t v) { return (v + 255) / 256 * 256; }

}  // namespace

cudaError_t launch_gptq_update(const sdq_plan_s* pl, float* W, const float* et, const float* U, int b,
                               cudaStream_t st) {
  const Geometry& g = pl->geo;
  const int f0 = b * g.block, col0 = f0 + g.block;
  if (col0 >= g.k_in) return cudaSuccess;
  const dim3 grid((g.k_in - col0 + kUpT - 1) / kUpT, (g.n_out + kUpT - 1) / kUpT);
  if (grid.y > 65535) return cudaErrorInvalidConfiguration;
  gptq_update_kernel<<<grid, kUpThreads, 0, st>>>(W, et, U, g.n_out, g.k_in, g.block, f0, col0);
  return cudaGetLastError();
}

}  // namespace sdq

using namespace sdq;

extern "C" size_t sdq_gptq_workspace_bytes(sdq_plan p) {
  if (!p) return 0;
  const Geometry& g = p->geo;
  return align256(sizeof(float) * (size_t)g.n_out * g.k_in) + align256(sizeof(float) * (size_t)g.n_out * g.block);
}

extern "C" int sdq_encode_rows_gptq(sdq_plan p, const float* W, const float* U, uint32_t* codes_plain,
                                    float* alpha, void* ws, size_t ws_bytes, void* stream) {
  if (!p || !W || !U || !codes_plain || !alpha || !ws) return SDQ_ERR_INVALID_ARG;
  const uintptr_t mis = (reinterpret_cast<uintptr_t>(W) | reinterpret_cast<uintptr_t>(U) |
                         reinterpret_cast<uintptr_t>(codes_plain) | reinterpret_cast<uintptr_t>(alpha) |
                         reinterpret_cast<uintptr_t>(ws)) & 15u;
  if (mis) return SDQ_ERR_INVALID_ARG;
  const Geometry& g = p->geo;
  if (g.block % 4) return SDQ_ERR_UNSUPPORTED;
  if (ws_bytes < sdq_gptq_workspace_bytes(p)) return SDQ_ERR_WORKSPACE;
  const int dv = sdq_check_device(p);
  if (dv != SDQ_OK) return dv;
  cudaStream_t st = (cudaStream_t)stream;
  float* wc = static_cast<float*>(ws);
  float* et = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + align256(sizeof(float) * (size_t)g.n_out * g.k_in));
  cudaError_t e = cudaMemcpyAsync(wc, W, sizeof(float) * (size_t)g.n_out * g.k_in, cudaMemcpyDeviceToDevice, st);
  // alpha from the original weights (pass 0 over every block)
  if (e == cudaSuccess) e = launch_encode_range(p, wc, codes_plain, alpha, st, 0, 1, 0, g.nblk, nullptr, nullptr);
  for (int b = 0; b < g.nblk && e == cudaSuccess; ++b) {
    e = launch_encode_range(p, wc, codes_plain, alpha, st, 1, 2, b, b + 1, U, et);
    if (e == cudaSuccess && b + 1 < g.nblk) e = launch_gptq_update(p, wc, et, U, b, st);
  }
  return e == cudaSuccess ? SDQ_OK : SDQ_ERR_CUDA;
}
