// coarse_tc.h -- group-key scores on the tensor cores (bf16 memories).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "htam.h"

namespace htam {

// s1[b][g] = q_b . (hi_g + lo_g) for b < B, g < G (-inf where count[g] == 0).
// queries [B, d] bf16; hi, lo [G, d] bf16 (the split fp32 group keys).
htam_status launch_coarse_tc(const void *queries, int B, int d, const __nv_bfloat16 *hi, const __nv_bfloat16 *lo,
                             const int32_t *count, int G, float *s1, unsigned *status, uint32_t max_polls,
                             cudaStream_t st);

}  // namespace htam
