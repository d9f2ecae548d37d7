// prefix.cu -- reduced queries of the prefix-attended lookup.
//
// The global-direction score of Eq. 9 sums the transition utility over the
// prefix of Eq. 8 with the position-aware weights of Eq. 10:
//   score(g) = sum_{i=1..P} alpha_i (q_i . c_g),  alpha_i = exp(-lambda (P - i)).
// The scorer is linear in the query, so score(g) = qbar . c_g with
// qbar = sum_i alpha_i q_i, and the whole lookup runs on qbar.  This kernel
// forms qbar: one thread per 8 consecutive elements of a query (one 16-byte
// load of bf16, two of fp32 per prefix element), fp32 accumulation over
// i = 1..P in order, one rounding to the memory's dtype at the end.  The
// weights come from the host (computed in double, passed as fp32).

#include "common.cuh"
#include "internal.h"

namespace htam {

namespace {

template <typename T>
__global__ void __launch_bounds__(256) prefix_reduce_kernel(const T *__restrict__ prefix, int32_t b, int32_t p_len,
                                                            int32_t d, PrefixWeights w, T *__restrict__ out) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int per_row = d / 8;
  if (t >= (int64_t)b * per_row) return;
  const int64_t q = t / per_row;
  const int j0 = (int)(t % per_row) * 8;
  float acc[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) acc[k] = 0.f;
  for (int i = 0; i < p_len; ++i) {
    const T *src = prefix + ((q * p_len + i) * d + j0);
    float x[8];
    if constexpr (sizeof(T) == 2) {
      const uint4 v = *reinterpret_cast<const uint4 *>(src);
      x[0] = bf16lo(v.x); x[1] = bf16hi(v.x); x[2] = bf16lo(v.y); x[3] = bf16hi(v.y);
      x[4] = bf16lo(v.z); x[5] = bf16hi(v.z); x[6] = bf16lo(v.w); x[7] = bf16hi(v.w);
    } else {
      const float4 a = *reinterpret_cast<const float4 *>(src);
      const float4 c = *reinterpret_cast<const float4 *>(src + 4);
      x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = c.x; x[5] = c.y; x[6] = c.z; x[7] = c.w;
    }
    const float alpha = w.alpha[i];
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[k] = fmaf(alpha, x[k], acc[k]);
  }
  T *dst = out + q * d + j0;
  if constexpr (sizeof(T) == 2) {
    uint32_t pk[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const __nv_bfloat162 h = __floats2bfloat162_rn(acc[2 * k], acc[2 * k + 1]);
      pk[k] = *reinterpret_cast<const uint32_t *>(&h);
    }
    *reinterpret_cast<uint4 *>(dst) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  } else {
    *reinterpret_cast<float4 *>(dst) = make_float4(acc[0], acc[1], acc[2], acc[3]);
    *reinterpret_cast<float4 *>(dst + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
}

}  // namespace

htam_status launch_prefix_reduce(const htam_memory *m, const void *prefix, int32_t b, int32_t p_len,
                                 const PrefixWeights &w, void *out, cudaStream_t st) {
  if (b == 0) return HTAM_OK;
  const int64_t threads = (int64_t)b * (m->d / 8);
  const unsigned blocks = (unsigned)ceil_div(threads, 256);
  if (m->dtype == HTAM_BF16) {
    launch_kernel(prefix_reduce_kernel<__nv_bfloat16>, blocks, 256, 0, st, static_cast<const __nv_bfloat16 *>(prefix), b,
                                                                 p_len, m->d, w, static_cast<__nv_bfloat16 *>(out));
  } else {
    launch_kernel(prefix_reduce_kernel<float>, blocks, 256, 0, st, static_cast<const float *>(prefix), b, p_len, m->d, w,
                                                        static_cast<float *>(out));
  }
  HTAM_CK_LAUNCH("prefix_reduce_kernel");
  return HTAM_OK;
}

}  // namespace htam
