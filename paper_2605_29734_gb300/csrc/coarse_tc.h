// coarse_tc.h -- group-key scores on the tensor cores (bf16 memories).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "htam.h"

namespace htam {

// K splits for B queries of dimension d against G groups on sm_count SMs:
// enough that the grid covers the SMs, at most one per 64-column K slice.
int coarse_tc_splits(int B, int d, int G, int sm_count);

// s1[z][b][g] = q_b[Kz] . (hi_g + lo_g)[Kz] for split z < splits (plane
// stride B * G), b < B, g < G (-inf where count[g] == 0), where Kz is split
// z's share of the 64-column K slices; the sum over z is q_b . (hi_g + lo_g).
// queries [B, d] bf16; hi, lo [G, d] bf16 (the split fp32 group keys).
// `splits` must be coarse_tc_splits(B, d, G, n) for some n (EINVAL otherwise).
// gate (device, may be NULL): when it points at a zero the kernel does
// nothing (a launch whose need is only known on the device).
htam_status launch_coarse_tc(const void *queries, int B, int d, const __nv_bfloat16 *hi, const __nv_bfloat16 *lo,
                             const int32_t *count, int G, int splits, float *s1, unsigned *status,
                             uint32_t max_polls, cudaStream_t st, const int32_t *gate = nullptr);

}  // namespace htam
