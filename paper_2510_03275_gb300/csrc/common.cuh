// Device helpers shared by the libsdq kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_fp8.h>
#include <cstdint>

#include "sdq_internal.h"

namespace sdq {

// ---------------------------------------------------------------- launches
DecodeConfig decode_config_search(const sdq_plan_s* plan, int M);
inline const DecodeConfig& decode_config(const sdq_plan_s* plan, int M) { return plan->dcfg[M]; }

struct WsLayout {
  size_t xt, pmax, frag, scale, part, cnt, err, total;
};
WsLayout workspace_layout(const sdq_plan_s* plan, int M);

// Kernel launchers (return cudaError_t of the launch).
cudaError_t launch_encode(const sdq_plan_s* p, const float* W, uint32_t* codes, float* alpha,
                          cudaStream_t st);
cudaError_t launch_pack(const sdq_plan_s* p, const uint32_t* plain, uint32_t* tiled, cudaStream_t st);
cudaError_t launch_unpack(const sdq_plan_s* p, const uint32_t* tiled, uint32_t* plain,
                          uint32_t* bad, cudaStream_t st);
cudaError_t launch_prep(const sdq_plan_s* p, const uint16_t* x, int M, void* ws, cudaStream_t st);
cudaError_t launch_decode(const sdq_plan_s* p, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st);
cudaError_t launch_prefill(const sdq_plan_s* p, const uint32_t* codes, const float* alpha, int M,
                           float* y, void* ws, cudaStream_t st);
cudaError_t launch_frag(const sdq_plan_s* p, int M, void* ws, cudaStream_t st);
int prep_partials(const sdq_plan_s* p, int M);  // per-row max partials of the prep grid
cudaError_t launch_read_prep(const sdq_plan_s* p, int M, const void* ws, float* out, cudaStream_t st);

// ------------------------------------------------------------------ device
__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
  return __uint_as_float((uint32_t)b << 16);
}

// Round-to-nearest-even fp32 -> bf16 bits (finite inputs).
__device__ __forceinline__ uint16_t float_to_bf16_bits(float f) {
  uint32_t u = __float_as_uint(f);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

// fp32 -> e4m3 byte (round to nearest even, saturating) and back.
__device__ __forceinline__ uint32_t f32_to_e4m3(float v) {
  __nv_fp8_e4m3 t(v);
  return (uint32_t)(*reinterpret_cast<const uint8_t*>(&t));
}
__device__ __forceinline__ float e4m3_to_f32(uint32_t b) {
  __nv_fp8_e4m3 t;
  *reinterpret_cast<uint8_t*>(&t) = (uint8_t)b;
  return (float)t;
}

// 16x8x32 warp MMA, e4m3 x e4m3 -> fp32.
__device__ __forceinline__ void mma_e4m3_16832(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 16x8x16 warp MMA, bf16 x bf16 -> fp32.
__device__ __forceinline__ void mma_bf16_16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}


// ------------------------------------------------- async copy / mbarrier
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(smem_u32(bar)),
               "r"(bytes) : "memory");
}
// 1-D bulk copy global -> shared (TMA), completion counted on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
          smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;\n" : "=l"(t));
  return t;
}
// Bounded wait for phase `parity` of `bar`: gives up after ~2 s of wall time
// and returns false (callers record an error and skip the dependent work).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  uint64_t t0 = 0;
  for (uint32_t i = 0;; ++i) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok) : "r"(a), "r"(parity) : "memory");
    if (ok) return true;
    if ((i & 1023u) == 0u) {
      const uint64_t now = globaltimer_ns();
      if (i == 0) t0 = now;
      else if (now - t0 > 2000000000ull) return false;
    }
  }
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}
// Programmatic dependent launch: wait for the preceding grid's completion
// (and memory), and allow the next grid in the stream to start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

// Launch with the programmatic-stream-serialization attribute, so that the
// kernel may begin while its predecessor in the stream finishes.
template <typename Kern, typename... Args>
cudaError_t launch_pdl(Kern k, dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, args...);
}

// Position of natural index kl (0..63) inside a 64-code stage of the prefill
// operand order: the order in which the prefill expander writes codes (and
// the prep kernel writes x_tilde) so that each 16-byte chunk of a bf16 tile
// row is one shift-and-mask expansion of a tiled word.
__host__ __device__ __forceinline__ int prefill_perm64(int kl) {
  const int qq = kl >> 5, r = kl & 31, h = r >> 4, t = (r & 15) >> 2, i = r & 3;
  const int inv = (i & 1) ? ((i >> 1) + 2 * h) : (4 + (i >> 1) + 2 * h);
  return 8 * (4 * qq + t) + inv;
}

}  // namespace sdq
