// common.cuh -- shared device/host helpers of the HTAM lookup library.
#pragma once

#include <atomic>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <climits>
#include <cmath>

#include "htam.h"

namespace htam {

constexpr int kPageRows = 128;       // entry rows per storage page
constexpr unsigned kFullMask = 0xffffffffu;
constexpr int kMaxK = 64;            // largest k_groups / k_entries

// Records the failing call for htam_last_error-style diagnostics.
void set_last_error(const char *what, cudaError_t err);

#define HTAM_CK(call)                                   \
  do {                                                  \
    cudaError_t err__ = (call);                         \
    if (err__ != cudaSuccess) {                         \
      ::htam::set_last_error(#call, err__);             \
      return HTAM_ECUDA;                                \
    }                                                   \
  } while (0)

#define HTAM_CK_LAUNCH(what)                            \
  do {                                                  \
    cudaError_t err__ = cudaGetLastError();             \
    if (err__ != cudaSuccess) {                         \
      ::htam::set_last_error(what, err__);              \
      return HTAM_ECUDA;                                \
    }                                                   \
  } while (0)

// ------------------------------------------------------------ element access
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// Low / high bf16 halves of a 32-bit word as fp32 (exact: a bf16 is the top
// 16 bits of the fp32 with the same value).
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// ------------------------------------------------------------ ordering
// Score descending, then id ascending (the tie rule of both levels).
__device__ __forceinline__ bool better(float a, int ia, float b, int ib) {
  return a > b || (a == b && ia < ib);
}

// A sorted list of up to 64 (score, id) pairs spread over one warp: lane l
// holds positions l (half 0) and l + 32 (half 1).  Empty slots hold
// (-inf, INT_MAX), worse than any real candidate.
struct WarpList {
  float s0, s1;
  int i0, i1;

  __device__ __forceinline__ void init() {
    s0 = s1 = -INFINITY;
    i0 = i1 = INT_MAX;
  }

  // The element at position k-1 (the admission threshold), broadcast.
  __device__ __forceinline__ void kth(int k, float &ts, int &ti) const {
    int pos = k - 1;
    int src = pos & 31;
    float a = __shfl_sync(kFullMask, pos < 32 ? s0 : s1, src);
    int b = __shfl_sync(kFullMask, pos < 32 ? i0 : i1, src);
    ts = a;
    ti = b;
  }

  // Merges a list sorted best first and held one pair per lane (lane t: the
  // t-th best) into slots 0..31; for k <= 32 only (slots 32..63 are not
  // touched).  The 32 best of two sorted lists A, B are better(A[i],
  // B[31-i]) for each i, a bitonic sequence, which five shuffle stages of
  // compare-and-exchange sort (better pair to the lower lane).
  __device__ __forceinline__ void merge32(float cs, int ci) {
    const int lane = threadIdx.x & 31;
    const float rs = __shfl_sync(kFullMask, cs, 31 - lane);
    const int ri = __shfl_sync(kFullMask, ci, 31 - lane);
    if (better(rs, ri, s0, i0)) {
      s0 = rs;
      i0 = ri;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ps = __shfl_xor_sync(kFullMask, s0, o);
      const int pi = __shfl_xor_sync(kFullMask, i0, o);
      const bool low = (lane & o) == 0;  // the lower lane of the pair keeps the better pair
      if (low == better(ps, pi, s0, i0)) {
        s0 = ps;
        i0 = pi;
      }
    }
  }

  // Inserts a warp-uniform candidate, keeping the 64 slots sorted.  All
  // lanes must call it with the same (s, id).
  __device__ __forceinline__ void insert(int k, float s, int id) {
    const int lane = threadIdx.x & 31;
    int p = __popc(__ballot_sync(kFullMask, better(s0, i0, s, id)));
    if (k > 32) p += __popc(__ballot_sync(kFullMask, better(s1, i1, s, id)));
    if (p >= k) return;
    float s0u = __shfl_up_sync(kFullMask, s0, 1);
    int i0u = __shfl_up_sync(kFullMask, i0, 1);
    float s1u = __shfl_up_sync(kFullMask, s1, 1);
    int i1u = __shfl_up_sync(kFullMask, i1, 1);
    float s31 = __shfl_sync(kFullMask, s0, 31);
    int i31 = __shfl_sync(kFullMask, i0, 31);
    if (lane == 0) {
      s1u = s31;
      i1u = i31;
    }
    if (lane > p) {
      s0 = s0u;
      i0 = i0u;
    } else if (lane == p) {
      s0 = s;
      i0 = id;
    }
    if (lane + 32 > p) {
      s1 = s1u;
      i1 = i1u;
    } else if (lane + 32 == p) {
      s1 = s;
      i1 = id;
    }
  }
};

// Sorts one (score, id) pair per lane across the warp, best first, with a
// bitonic network of shuffle compare-and-exchange stages.
__device__ __forceinline__ void warp_sort32(float &s, int &i) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
    for (int o = k >> 1; o > 0; o >>= 1) {
      const float ps = __shfl_xor_sync(kFullMask, s, o);
      const int pi = __shfl_xor_sync(kFullMask, i, o);
      const bool desc = (lane & k) == 0;  // this k-block ends up best first
      const bool low = (lane & o) == 0;
      if ((low == desc) == better(ps, pi, s, i)) {
        s = ps;
        i = pi;
      }
    }
  }
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFullMask, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFullMask, v, o);
  return v;
}

__host__ __device__ inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// ------------------------------------------------ programmatic dependent launch
// The kernels of a query (and of an append) run back to back on one stream.
// Launched with programmatic stream serialisation, a kernel's blocks may be
// scheduled while the previous kernel is still finishing; every kernel of
// those paths therefore starts with griddepcontrol.wait (returns once the
// previous kernel has completed and its writes are visible; a no-op when the
// launch had no programmatic dependency) before it touches device memory,
// and then lets its own dependents start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_entry() {
  pdl_wait();
  pdl_trigger();
}

// Whether the launches made by this host thread use programmatic stream
// serialisation (set for the duration of a query or append from the memory
// object's tuning).
extern thread_local bool g_launch_pdl;
struct PdlScope {
  bool prev;
  explicit PdlScope(bool on) : prev(g_launch_pdl) { g_launch_pdl = on; }
  ~PdlScope() { g_launch_pdl = prev; }
};

template <typename... P, typename... A>
inline cudaError_t launch_kernel(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                 A &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  if (g_launch_pdl) {
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
  }
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<A &&>(args)...);
}

// Launches `kernel` (parenthesise template kernels) and returns HTAM_ECUDA
// from the enclosing function if the launch fails.
#define HTAM_LAUNCH(what, kernel, grid, block, smem, st, ...)                                   \
  do {                                                                                        \
    cudaError_t err__ = ::htam::launch_kernel(kernel, dim3(grid), dim3(block), (size_t)(smem), \
                                              st, __VA_ARGS__);                               \
    if (err__ != cudaSuccess) {                                                               \
      ::htam::set_last_error(what, err__);                                                    \
      return HTAM_ECUDA;                                                                      \
    }                                                                                         \
  } while (0)

// True the first time it is called for the current device with this flag
// word (one bit per device): per-device, once-only setup such as a kernel's
// shared-memory limit, safe to call from several host threads.
inline bool first_on_device(std::atomic<uint64_t> &done) {
  int dev = 0;
  cudaGetDevice(&dev);
  const uint64_t bit = uint64_t(1) << (dev & 63);
  return (done.fetch_or(bit) & bit) == 0;
}

}  // namespace htam
