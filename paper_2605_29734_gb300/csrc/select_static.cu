// select_static.cu -- group selection that allocates nothing.
//
// htam_select_groups_static computes the same group selection as the first
// stage of htam_query (coarse scores q . c_g against every group key, then the
// k_groups best), but its only scratch -- the [b, n_groups] fp32 score matrix
// -- lives in a fixed array compiled into the library instead of scratch the
// memory object grows with cudaMalloc.
//
// Who needs this: callers that must not allocate device memory while they
// serve requests -- a server whose device memory is fully reserved up front
// (an allocation could fail or fragment the pool), code running inside an
// allocator callback or a memory-pool owner that would re-enter itself, and
// latency-critical loops that cannot take the implicit device-wide
// synchronisation that cudaFree performs.
//
// The array is HTAM_STATIC_SCRATCH_BYTES (16 MiB) of device memory that every
// GPU which loads the library keeps until the process exits.  All calls share
// it and it keeps the previous call's contents: every call writes the part it
// later reads, so nothing has to start at zero, but two calls whose work
// overlaps on the GPU (different streams, or different host threads) race on
// it and must be serialised by the caller.

#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace htam {

namespace {

constexpr size_t kStaticFloats = HTAM_STATIC_SCRATCH_BYTES / sizeof(float);

// The scratch.  Host code must not pass this symbol to a kernel (on the host
// it names a host-side stand-in, not device memory): its device address is
// looked up once per device with cudaGetSymbolAddress.
static __device__ __align__(256) float g_static_scores[kStaticFloats];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
float *g_scores_addr[kMaxDevices] = {};

// Device address of the scratch on `device` (which must be current).
htam_status static_scores_on(int device, float **out) {
  if (device < 0 || device >= kMaxDevices) return HTAM_EINVAL;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scores_addr[device]) {
    void *p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_static_scores);
    if (e != cudaSuccess) {
      set_last_error("cudaGetSymbolAddress(g_static_scores)", e);
      return HTAM_ECUDA;
    }
    g_scores_addr[device] = static_cast<float *>(p);
  }
  *out = g_scores_addr[device];
  return HTAM_OK;
}

// s1[b][g] = q_b . cent_g, each output accumulated with fmaf over k = 0..d-1
// in order against the fp32 group key (htam_query reaches the same scores
// within fp32 rounding, on the tensor cores for bf16 memories); -inf for empty
// groups.  32x32 tiles: query tiles on grid.x (up to 2^31 - 1 blocks), group
// tiles on grid.y (at most 2,048 for 65,536 groups).
template <typename T>
__global__ void __launch_bounds__(256) static_coarse_kernel(const T *__restrict__ Q, int B, int d,
                                                            const float *__restrict__ cent,
                                                            const int32_t *__restrict__ count, int G,
                                                            float *__restrict__ s1) {
  __shared__ float qs[32][33];
  __shared__ float cs[32][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8 threads
  const int b0 = blockIdx.x * 32, g0 = blockIdx.y * 32;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int k0 = 0; k0 < d; k0 += 32) {
    for (int r = ty; r < 32; r += 8) {
      int k = k0 + tx;
      qs[r][tx] = (b0 + r < B && k < d) ? to_f32(Q[(int64_t)(b0 + r) * d + k]) : 0.f;
      cs[r][tx] = (g0 + r < G && k < d) ? cent[(int64_t)(g0 + r) * d + k] : 0.f;
    }
    __syncthreads();
    for (int k = 0; k < 32; ++k) {  // zero padding past d, as in htam_query
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[i] = fmaf(qs[ty + 8 * i][k], cs[tx][k], acc[i]);
    }
    __syncthreads();
  }
  const int g = g0 + tx;
  if (g >= G) return;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int b = b0 + ty + 8 * i;
    if (b < B) s1[(int64_t)b * G + g] = count[g] > 0 ? acc[i] : -INFINITY;
  }
}

// One warp per query: the k_groups best groups (score descending, lower id
// on ties, empty groups excluded, -1 / -inf padding).
__global__ void static_select_kernel(const float *__restrict__ s1, int B, int G,
                                     const int32_t *__restrict__ count, int kg,
                                     int32_t *__restrict__ gidx, float *__restrict__ gscore) {
  int b = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (b >= B) return;
  WarpList L;
  L.init();
  float ts = -INFINITY;
  int ti = INT_MAX;
  for (int g0 = 0; g0 < G; g0 += 32) {
    int g = g0 + lane;
    bool valid = g < G && count[g] > 0;
    float s = valid ? s1[(int64_t)b * G + g] : -INFINITY;
    unsigned mask = __ballot_sync(kFullMask, valid && better(s, g, ts, ti));
    while (mask) {
      int src = __ffs(mask) - 1;
      mask &= mask - 1;
      L.insert(kg, __shfl_sync(kFullMask, s, src), g0 + src);
      L.kth(kg, ts, ti);
    }
  }
  if (lane < kg) {
    gidx[(int64_t)b * kg + lane] = L.i0 == INT_MAX ? -1 : L.i0;
    gscore[(int64_t)b * kg + lane] = L.i0 == INT_MAX ? -INFINITY : L.s0;
  }
  if (lane + 32 < kg) {
    gidx[(int64_t)b * kg + lane + 32] = L.i1 == INT_MAX ? -1 : L.i1;
    gscore[(int64_t)b * kg + lane + 32] = L.i1 == INT_MAX ? -INFINITY : L.s1;
  }
}

}  // namespace

}  // namespace htam

using namespace htam;

extern "C" htam_status htam_select_groups_static(const htam_memory *m, const void *queries, int32_t b,
                                                 int32_t k_groups, int32_t *group_idx, float *group_score,
                                                 void *cuda_stream) {
  if (!m || b < 0 || b > (1 << 24) || k_groups < 1 || k_groups > kMaxK || k_groups > m->n_groups) {
    return HTAM_EINVAL;
  }
  if (b == 0) return HTAM_OK;
  if (!queries || !group_idx || !group_score) return HTAM_EINVAL;
  if ((reinterpret_cast<uintptr_t>(queries) & 15u) != 0) return HTAM_EINVAL;
  // The score matrix must fit the fixed scratch.
  if ((uint64_t)b * (uint64_t)m->n_groups > kStaticFloats) return HTAM_EINVAL;
  int device = -1;
  HTAM_CK(cudaGetDevice(&device));
  if (device != m->device) return HTAM_EINVAL;
  float *s1 = nullptr;
  htam_status s = static_scores_on(device, &s1);
  if (s != HTAM_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const int G = m->n_groups, d = m->d;
  // b <= 2^24 gives at most 2^19 query tiles on grid.x and G <= 65,536 at
  // most 2,048 group tiles on grid.y: both within the launch limits, so no
  // argument that passed the checks above fails at launch.
  dim3 grid((unsigned)ceil_div(b, 32), (unsigned)ceil_div(G, 32));
  if (m->dtype == HTAM_BF16) {
    static_coarse_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(static_cast<const __nv_bfloat16 *>(queries), b, d,
                                                              m->cent, m->count, G, s1);
  } else {
    static_coarse_kernel<float><<<grid, 256, 0, st>>>(static_cast<const float *>(queries), b, d, m->cent,
                                                      m->count, G, s1);
  }
  HTAM_CK_LAUNCH("static_coarse_kernel");
  static_select_kernel<<<(unsigned)ceil_div((int64_t)b * 32, 256), 256, 0, st>>>(s1, b, G, m->count, k_groups,
                                                                                 group_idx, group_score);
  HTAM_CK_LAUNCH("static_select_kernel");
  return HTAM_OK;
}
