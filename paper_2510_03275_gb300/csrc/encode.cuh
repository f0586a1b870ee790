// Launchers of the encoder's block-range form and of the GPTQ update (used by
// the encoder with GPTQ block compensation).  Internal to libsdq.
#pragma once

#include "common.cuh"

namespace sdq {

// Passes [pass0, pass1) (0: alpha, 1: scan) over blocks [b0, b1); with `et`
// non-null, pass 1 also writes each block's normalised GPTQ error (n_out x B)
// using the factor U (k_in x k_in).
cudaError_t launch_encode_range(const sdq_plan_s* p, const float* W, uint32_t* codes, float* alpha,
                                cudaStream_t st, int pass0, int pass1, int b0, int b1, const float* U,
                                float* et);
// W[:, col0:] -= E~ U[b B : (b + 1) B, col0:] (col0 = (b + 1) B) in the canonical order.
cudaError_t launch_gptq_update(const sdq_plan_s* p, float* W, const float* et, const float* U, int b,
                               cudaStream_t st);

}  // namespace sdq
