// Device helpers shared by the libsdq kernels (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <atomic>
#include <cstdint>

#include "sdq_internal.h"

namespace sdq {

// ---------------------------------------------------------------- launches
DecodeConfig decode_config_search(const sdq_plan_s* plan, int M);
inline const DecodeConfig& decode_config(const sdq_plan_s* plan, int M) { return plan->dcfg[M]; }

// Workspace regions (byte offsets).  cnt: one 64-bit split-K ticket per row
// tile; err: the call record (two 64-bit words, see call_record_*).
struct WsLayout {
  size_t xt, bimg, sfbw, part, cnt, err, total;
  size_t what;   // rebuilt weights W' (n_out x k_in bf16) of the dense large-batch route
};
WsLayout workspace_layout(const sdq_plan_s* plan, int M);
// SDQ_OK when the current device is the plan's, else SDQ_ERR_INVALID_ARG (or
// SDQ_ERR_CUDA).
int sdq_check_device(const sdq_plan_s* p);
// SDQ_ERR_TIMEOUT when the call record in `ws` (layout of plan p, batch M)
// says the last call gave up a bounded wait, else SDQ_OK; synchronizes
// `stream`.
int workspace_record_status(const sdq_plan_s* p, int32_t M, const void* ws, void* stream);
// Number of a contraction call, from one process-wide counter (never 0).
uint64_t next_call_number();
// Tag of call number n for the workspace's tickets and call record: a
// bijection of the low 47 bits of n, scrambled, with bit 47 set (48 bits).
uint64_t call_tag(uint64_t n);

// Kernel launchers (return cudaError_t of the launch).
cudaError_t launch_encode(const sdq_plan_s* p, const float* W, uint32_t* codes, float* alpha,
                          cudaStream_t st);
cudaError_t launch_pack(const sdq_plan_s* p, const uint32_t* plain, uint32_t* tiled, cudaStream_t st);
cudaError_t launch_unpack(const sdq_plan_s* p, const uint32_t* tiled, uint32_t* plain,
                          uint32_t* bad, cudaStream_t st);
// y_zero (M x n_out, may be null): cleared by the decode prepare kernel.
cudaError_t launch_prep(const sdq_plan_s* p, const uint16_t* x, int M, void* ws, cudaStream_t st,
                        float* y_zero = nullptr);
// The dense large-batch route (rebuild W' = 2 C G, then y = alpha / 2 W' x):
// whether it applies to plan p at batch M, and its two launches.
bool dense_route_applies(const sdq_plan_s* p, int M);
cudaError_t launch_dense_forward(const sdq_plan_s* p, const uint32_t* codes, const float* alpha,
                                 const uint16_t* x, int M, float* y, void* ws, cudaStream_t st);
// cuTensorMapEncodeTiled from the driver (null if unavailable), as void*.
void* tensor_map_encoder();
// Prefill prepare (M > 64) on the tensor cores where the layer allows it;
// *used = false (nothing launched) otherwise.
cudaError_t launch_prep_tc(const sdq_plan_s* p, const uint16_t* x, int M, void* ws, cudaStream_t st,
                           bool* used);
// early = 1: the decode kernel starts streaming codes before waiting for the
// preceding grid (valid only behind this library's own prep kernels).
// y_mode: kYStore: y = the result (split-K by the deterministic ticket
// route); kYZeroed: y holds zeros (the prepare kernel of the same call
// cleared it), so that split-K partial sums are added into it by float
// reductions (order of the additions not fixed); kYAdd: y += the result, by
// float reductions whatever the split.
constexpr int kYStore = 0, kYZeroed = 1, kYAdd = 2;
cudaError_t launch_decode(const sdq_plan_s* p, const uint32_t* codes, const float* alpha, int M,
                          float* y, void* ws, cudaStream_t st, int early, int y_mode);
// Whether the decode prepare kernel writes the B operand image (n_b a
// multiple of 64), so that each decode CTA copies its chunk's part.
bool decode_image(const sdq_plan_s* p);
cudaError_t launch_prefill(const sdq_plan_s* p, const uint32_t* codes, const float* alpha, int M,
                           float* y, void* ws, cudaStream_t st);
cudaError_t launch_read_prep(const sdq_plan_s* p, int M, const void* ws, float* out, cudaStream_t st);

// Raise `kernel`'s dynamic shared-memory limit to `bytes` once per device:
// the setting is per function and device, and a constant value makes later
// launches (and concurrent callers) skip the driver call.
template <class Kern>
cudaError_t smem_limit_once(Kern kernel, int bytes, int device, std::atomic<int>* done) {
  if (device >= 0 && device < 64 && done[device].load(std::memory_order_acquire)) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && device >= 0 && device < 64) done[device].store(1, std::memory_order_release);
  return e;
}

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

// Two fp32 -> bf16 (round to nearest even), lo in bits 0-15, hi in 16-31.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;\n" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
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
// The same, with an L2 eviction-priority hint (data read once, e.g. decode
// code streams: evict them first so that small reused tables stay in L2).
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ void bulk_g2s_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                              uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;\n"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy) : "memory");
}
// Bounded wait for phase `parity` of `bar`: gives up after ~4e9 SM cycles
// (about 2 s) and returns false (callers record an error and skip the
// dependent work).  The clock is read only once the first test has failed.
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(a), "r"(parity) : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  if (mbar_try(a, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try(a, parity))
    if (clock64() - t0 > 4000000000ll) return false;
  return true;
}
// 16-byte global -> shared copy that does not pass through registers (`bytes`
// = 0 fills the destination with zeros); completion by cp_async_wait_all.
__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n"
               :: "r"(smem_u32(dst)), "l"(src), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
// Fire-and-forget float add into global memory (no value returned, so the
// issuing thread does not wait for the round trip).
__device__ __forceinline__ void red_add_f32(float* addr, float v) {
  asm volatile("red.relaxed.gpu.global.add.f32 [%0], %1;\n" :: "l"(addr), "f"(v) : "memory");
}
// 4-byte global -> shared copy (cp.async group semantics as above).
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" :: "r"(smem_u32(dst)), "l"(src) : "memory");
}
// Wait until at most N of this thread's cp.async groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
  asm volatile("cp.async.wait_group %0;\n" :: "n"(N) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;\n" ::: "memory");
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

// ------------------------------------------------------ tcgen05 / TMEM
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(dst)),
               "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate) : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                   smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar)) : "memory");
}
// 32 TMEM lanes x 16 columns of 32-bit values: register i of the thread of
// lane l holds (lane base + l, column + i).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
      " [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
                 "=r"(r[7])
               : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (SBO), start address in 16-byte units.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                 // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;       // stride byte offset
  d |= (uint64_t)1 << 46;                 // descriptor version
  d |= (uint64_t)2 << 61;                 // SWIZZLE_128B
  return d;
}

// 32 TMEM lanes x 16 (8) columns of 32-bit values from registers: register
// i of the thread of lane l goes to (lane base + l, column + i).
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n"
      ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]) : "memory");
}
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};\n" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]) : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
      "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
      "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st4(uint32_t taddr, const uint32_t (&r)[4]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(taddr), "r"(r[0]), "r"(r[1]),
               "r"(r[2]), "r"(r[3]) : "memory");
}
__device__ __forceinline__ void tmem_st1(uint32_t taddr, uint32_t v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};\n" ::"r"(taddr), "r"(v) : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory"); }

// D (TMEM, fp32) (+)= A (TMEM, e2m1) . B (smem descriptor, e2m1)^T, M = 128,
// K = 64, with the block scales of A and B read from TMEM (one ue8m0 scale
// per 32 K; this library stores 1.0 everywhere and scales in the epilogue).
// A in TMEM: lane = row, column c nibble i (low first) = K index 8 c + i.
// B in shared memory: K-major, byte j nibble h (low first) = K index 2 j + h.
__device__ __forceinline__ void umma_mxf4_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                             uint32_t sfa_tmem, uint32_t sfb_tmem, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %6, 0;\n"
      " tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], [%1], %2, %3, [%4], [%5], p;\n}\n"
      ::"r"(d_tmem), "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(sfa_tmem), "r"(sfb_tmem), "r"(accumulate)
      : "memory");
}
// Instruction descriptor of umma_mxf4_ts: A and B e2m1, ue8m0 scales,
// M = 128, N = n (a multiple of 16, at most 256), dense, both K-major.
__host__ __device__ constexpr uint32_t mxf4_idesc(int n) {
  return (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | (1u << 23) | (1u << 27);
}
// ue8m0 1.0 in every byte of a scale-factor column.
constexpr uint32_t kUnitScales = 0x7F7F7F7Fu;

// Two fp32 values to a byte of e2m1 codes (round to nearest even, saturating
// at +-6): `lo` in bits 0-3, `hi` in bits 4-7; `q` receives the two values
// the codes stand for (exact).
__device__ __forceinline__ uint32_t e2m1x2(float lo, float hi, float2* q) {
  uint16_t b;
  uint32_t h2;
  asm("{\n .reg .b8 t;\n cvt.rn.satfinite.e2m1x2.f32 t, %3, %2;\n mov.b16 %0, {t, 0};\n"
      " cvt.rn.f16x2.e2m1x2 %1, t;\n}\n"
      : "=h"(b), "=r"(h2) : "f"(lo), "f"(hi));
  *q = __half22float2(*reinterpret_cast<const __half2*>(&h2));
  return b;
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;\n" ::"r"(id), "r"(nthreads) : "memory");
}

// Call record in the workspace: word 0 = tag of the last call that gave up a
// bounded wait, word 1 = tag of the last call that ran.  Tags (call_tag in
// capi.cu) are 48-bit values with bit 47 set, distinct for 2^47 calls and
// scrambled, so that neither zeroed memory nor structured leftovers of
// another call, plan or batch size (counters, small floats) read as the
// current call's: nothing in the workspace needs resetting.
__device__ __forceinline__ void call_record_start(uint64_t* rec, uint64_t call, bool leader) {
  if (leader) rec[1] = call;
}
__device__ __forceinline__ void call_record_fail(uint64_t* rec, uint64_t call) {
  atomicExch(reinterpret_cast<unsigned long long*>(rec), (unsigned long long)call);
}

__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;\n" ::: "memory"); }

// Split-K ticket of one row tile: bits 16..63 the call's tag, bits 0..15 the
// arrivals of that call.  A ticket that carries another tag counts as empty.
// One acq_rel fence (after the CTA barrier that orders the other threads'
// partial stores before it) publishes the CTA's partials; then every arrival
// adds 1, and an add that found another tag installs (tag, 1) by
// compare-and-swap or joins the call that another arrival installed
// meanwhile.  (Such adds never carry into the tag field: a call leaves at
// most 2 S arrivals in a ticket, far below 2^16.)  The last arrival
// (n == total) fences again before reading the other CTAs' partials and
// clears the ticket, so that a workspace that is only ever used for these
// calls keeps zeros there.  Returns this CTA's arrival number (1..total), or
// 0 if the compare-and-swap did not settle within its retry bound.
__device__ __forceinline__ uint32_t ticket_take(uint64_t* tk, uint64_t call, uint32_t total) {
  unsigned long long* p = reinterpret_cast<unsigned long long*>(tk);
  fence_acq_rel_gpu();
  const unsigned long long old = atomicAdd(p, 1ull);
  uint32_t n = 0;
  if ((old >> 16) == call) {
    n = (uint32_t)(old & 0xFFFFu) + 1;
  } else {
    unsigned long long cur = old + 1;   // another call's ticket, with our add in it
    for (int it = 0; it < 64 && n == 0; ++it) {
      const unsigned long long prev = atomicCAS(p, cur, (call << 16) | 1ull);
      if (prev == cur) n = 1;
      else if ((prev >> 16) == call) n = (uint32_t)(atomicAdd(p, 1ull) & 0xFFFFu) + 1;
      else cur = prev;
    }
  }
  if (n == total) {
    fence_acq_rel_gpu();
    atomicExch(p, 0ull);
  }
  return n;
}

// Install `call`'s tag in a ticket ahead of the arrivals (count 0), unless
// an arrival already did: one read and at most one compare-and-swap, issued
// at kernel start so that the end-of-kernel arrivals find the tag and take
// the one-atomic path of ticket_take.  A lost race is harmless: ticket_take
// installs or joins the tag itself.
__device__ __forceinline__ void ticket_install(uint64_t* tk, uint64_t call) {
  unsigned long long* p = reinterpret_cast<unsigned long long*>(tk);
  const unsigned long long old = *reinterpret_cast<volatile unsigned long long*>(p);
  if ((old >> 16) != call) atomicCAS(p, old, call << 16);
}

// MMA K position kap (within a 128-code block) of natural code kl: the
// inverse of decode_stage_k.
//   ternary: kl = 16 w + 2 n + s -> kap = 16 w + 8 s + n
//   binary:  kl = 32 w + 4 n + k -> kap = 32 w + 8 k + n
__host__ __device__ __forceinline__ int decode_pos(int kl, bool ternary) {
  if (ternary) {
    const int f = kl & 15;
    return (kl & ~15) + 8 * (f & 1) + (f >> 1);
  }
  const int f = kl & 31;
  return (kl & ~31) + 8 * (f & 3) + (f >> 2);
}

// Natural k (within a 128-code decode block) at MMA K index kap = 8 c + n
// (TMEM column c of the block's 16, nibble n): the order in which the decode
// expander turns a row's packed words into e2m1 nibbles.
//   ternary: word w (codes 16 w .. 16 w + 15, 2 bits each) gives column 2 w
//            (even codes: nibble n = code 16 w + 2 n) and column 2 w + 1
//            (odd codes: nibble n = code 16 w + 2 n + 1)
//   binary:  word w (codes 32 w .. 32 w + 31) gives columns 4 w + k, k < 4,
//            nibble n = code 32 w + 4 n + k
__host__ __device__ __forceinline__ int decode_stage_k(int kap, bool ternary) {
  if (ternary) {
    const int kp = kap & 15;
    return (kap & ~15) + 2 * (kp & 7) + (kp >> 3);
  }
  const int kp = kap & 31;
  return (kap & ~31) + 4 * (kp & 7) + (kp >> 3);
}

// Position of natural index kl (0..63) inside a 64-code stage of the prefill
// operand order: the order in which the prefill expander writes a row's codes
// (and the prep kernel writes x_tilde) when word i of the row is expanded by
// shift-and-mask into bf16 pairs.
//   ternary: pair j of word i (i < 4, j < 8) holds codes 16i + 7 - j (low
//            half) and 16i + 15 - j (high half) at positions 16i + 2j, +1
//   binary:  pair j of word i (i < 2, j < 16) holds codes 32i + 15 - j and
//            32i + 31 - j at positions 32i + 2j, +1
__host__ __device__ __forceinline__ int prefill_pos64(int kl, bool ternary) {
  if (ternary) {
    const int i = kl >> 4, f = kl & 15;
    return f < 8 ? 16 * i + 2 * (7 - f) : 16 * i + 2 * (15 - f) + 1;
  }
  const int i = kl >> 5, f = kl & 31;
  return f < 16 ? 32 * i + 2 * (15 - f) : 32 * i + 2 * (31 - f) + 1;
}

}  // namespace sdq
