// K5: prefill contraction (M > 64) on the 5th-generation tensor cores.
// Placeholder until the tcgen05 kernel lands: reports "not supported".
#include "common.cuh"

namespace sdq {

cudaError_t launch_prefill(const sdq_plan_s*, const uint32_t*, const float*, int, float*, void*,
                           cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace sdq
