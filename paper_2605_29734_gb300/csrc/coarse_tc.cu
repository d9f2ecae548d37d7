// coarse_tc.cu -- group-key scores on the tcgen05 tensor cores.
//
// s1[b][g] = q_b . c_g (Eq. 9 with the linear scorer of App. B.6) for a bf16
// memory.  The key c_g is the fp32 mean of group g's entries; it enters the
// MMA as the sum of two bf16 matrices, hi = bf16(c) and lo = bf16(c - hi),
// so that q . hi + q . lo carries the key to about 2^-17 of its size while
// both operands stay bf16 (the query itself is bf16 already).  Each CTA owns
// one 128-query x 128-group tile (two CTAs per SM): TMA stages 64-column K slices of Q, hi and
// lo (128-byte swizzle), one thread issues per slice four MMAs against hi and
// four against lo into the same fp32 accumulator in tensor memory, and four
// epilogue warps write the scores (-inf for empty groups) for the top-k
// kernel, turned around in shared memory so that each store covers a
// 128-byte row segment.  When the tiles alone would leave SMs idle (few queries), the K
// slices are split over blockIdx.z: split z writes its partial dot products
// to plane z of the output, and the top-k kernel adds the planes in order.
// Every mbarrier wait is bounded.

#include <algorithm>

#include "coarse_tc.h"
#include "common.cuh"
#include "fine_tc.h"
#include "sm100.cuh"

namespace htam {

namespace {

using namespace sm100;

constexpr int kCStages = 2;
constexpr int kCKBlock = 64;
constexpr int kCM = 128;                           // queries per tile (MMA M)
constexpr int kCN = 128;                           // groups per tile (MMA N): one page of keys
constexpr int kCABytes = kCM * kCKBlock * 2;       // 16 KiB
constexpr int kCBBytes = kCN * kCKBlock * 2;       // 16 KiB (hi or lo)
constexpr int kCPerSM = 2;                         // CTAs resident per SM (96 KiB of stages each)
constexpr int kCThreads = 192;

struct __align__(8) CoarseBars {
  uint64_t full[kCStages];
  uint64_t empty[kCStages];
  uint64_t acc_full;
  uint32_t tmem_base;
  int abort;
};

constexpr size_t kCSmem = 1024 + kCStages * (kCABytes + 2 * kCBBytes) + sizeof(CoarseBars);

__global__ void __launch_bounds__(kCThreads, kCPerSM)
    coarse_tc_kernel(const __grid_constant__ CUtensorMap q_map, const __grid_constant__ CUtensorMap hi_map,
                     const __grid_constant__ CUtensorMap lo_map, int d, int kb_per, const int32_t *__restrict__ count,
                     int B, int G, float *__restrict__ s1, unsigned *status, uint32_t max_polls,
                     const int32_t *__restrict__ gate) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  // Gated launch (rows appended without a group): nothing to score.  The
  // exit is uniform over the grid and comes before any barrier or tensor
  // memory is set up.
  if (gate && *gate == 0) return;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t *smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
  uint8_t *st_a = smem;
  uint8_t *st_hi = st_a + kCStages * kCABytes;
  uint8_t *st_lo = st_hi + kCStages * kCBBytes;
  CoarseBars *sh = reinterpret_cast<CoarseBars *>(st_lo + kCStages * kCBBytes);
  volatile int *abort = &sh->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * kCM, n0 = blockIdx.y * kCN;
  const int nk_all = (d + kCKBlock - 1) / kCKBlock;
  const int kb0 = blockIdx.z * kb_per;                // this split's K slices: [kb0, kb0 + nk)
  const int nk = min(nk_all, kb0 + kb_per) - kb0;     // >= 1 by the launch
  s1 += (int64_t)blockIdx.z * B * G;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kCStages; ++s) {
      mbar_init(&sh->full[s], 1);
      mbar_init(&sh->empty[s], 1);
    }
    mbar_init(&sh->acc_full, 1);
    sh->abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(&sh->tmem_base, kCN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = sh->tmem_base;
  bool ok = true;

  if (warp == 0) {
    uint32_t ph = 0;
    int st = 0;
    for (int kb = 0; kb < nk; ++kb) {
      if (!mbar_wait(&sh->empty[st], ph ^ 1u, abort, max_polls)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        const uint32_t bytes = kCABytes + 2u * kCBBytes;
        mbar_arrive_expect_tx(&sh->full[st], bytes);
        const int x = (kb0 + kb) * kCKBlock;
        tma_load_2d(smem_addr(st_a + st * kCABytes), &q_map, x, m0, &sh->full[st]);
        tma_load_2d(smem_addr(st_hi + st * kCBBytes), &hi_map, x, n0, &sh->full[st]);
        tma_load_2d(smem_addr(st_lo + st * kCBBytes), &lo_map, x, n0, &sh->full[st]);
      }
      __syncwarp();
      if (++st == kCStages) {
        st = 0;
        ph ^= 1u;
      }
    }
    // Drain: the last stages' copies have landed.
    for (int back = 1; back <= kCStages && back <= nk; ++back) {
      const int kb = nk - back;
      for (uint32_t i = 0; i < max_polls && !mbar_try_wait(&sh->full[kb % kCStages], (kb / kCStages) & 1u); ++i) {
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    const uint32_t idesc = idesc_bf16_f32(kCM, kCN);
    uint32_t ph = 0;
    int st = 0;
    for (int kb = 0; kb < nk; ++kb) {
      if (!mbar_wait(&sh->full[st], ph, abort, max_polls)) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (lane == 0) {
        const uint64_t ad = sw128_kmajor_desc(smem_addr(st_a + st * kCABytes));
        const uint64_t hd = sw128_kmajor_desc(smem_addr(st_hi + st * kCBBytes));
        const uint64_t ld = sw128_kmajor_desc(smem_addr(st_lo + st * kCBBytes));
#pragma unroll
        for (int k = 0; k < kCKBlock / 16; ++k) umma_bf16(tbase, ad + 2 * k, hd + 2 * k, idesc, (kb | k) != 0);
#pragma unroll
        for (int k = 0; k < kCKBlock / 16; ++k) umma_bf16(tbase, ad + 2 * k, ld + 2 * k, idesc, 1u);
        umma_commit(&sh->empty[st]);
      }
      __syncwarp();
      if (++st == kCStages) {
        st = 0;
        ph ^= 1u;
      }
    }
    if (lane == 0) umma_commit(&sh->acc_full);  // also drains: arrives once every MMA is done
    __syncwarp();
  } else {
    const int quad = warp & 3;
    if (!mbar_wait(&sh->acc_full, 0, abort, max_polls)) ok = false;
    tc_fence_after();
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the stages' async-proxy use is over
    if (ok) {
      // Every MMA is done, so the operand stages are free: each warp turns
      // its 32 rows x 32 columns around in a padded shared-memory square and
      // writes whole 128-byte row segments (one per store instruction).
      float *sq = reinterpret_cast<float *>(smem) + (warp - 2) * 32 * 33;
      const int row0 = m0 + quad * 32;
      const uint32_t lane_addr = tbase + (static_cast<uint32_t>(quad * 32) << 16);
      for (int ch = 0; ch < kCN / 32; ++ch) {
        const int g0 = n0 + ch * 32;
        if (g0 >= G) break;  // uniform
        uint32_t r[32];
        __syncwarp();
        tmem_ld32(lane_addr + ch * 32, r);
        tmem_wait_ld(r);
#pragma unroll
        for (int j = 0; j < 32; ++j) sq[lane * 33 + j] = __uint_as_float(r[j]);
        __syncwarp();
        const int g = g0 + lane;
        const bool gin = g < G;
        const bool empty = !gin || count[g] == 0;
        for (int i = 0; i < 32 && row0 + i < B; ++i) {
          if (gin) s1[(int64_t)(row0 + i) * G + g] = empty ? -INFINITY : sq[i * 33 + lane];
        }
        __syncwarp();
      }
    }
  }
  if (!ok) {
    atomicOr(status, 1u);
    sh->abort = 1;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tbase, kCN);
  }
}

}  // namespace

int coarse_tc_splits(int B, int d, int G, int sm_count) {
  const int64_t tiles = ceil_div((int64_t)B, kCM) * ceil_div((int64_t)G, kCN);
  const int nk = (int)ceil_div((int64_t)d, kCKBlock);
  const int want =
      (int)std::max<int64_t>(1, std::min<int64_t>(nk, kCPerSM * sm_count / std::max<int64_t>(1, tiles)));
  const int kb_per = (int)ceil_div((int64_t)nk, want);
  return (int)ceil_div((int64_t)nk, kb_per);
}

htam_status launch_coarse_tc(const void *queries, int B, int d, const __nv_bfloat16 *hi, const __nv_bfloat16 *lo,
                             const int32_t *count, int G, int splits, float *s1, unsigned *status,
                             uint32_t max_polls, cudaStream_t st, const int32_t *gate) {
  CUtensorMap q_map, hi_map, lo_map;
  htam_status s = make_bf16_tile_map(&q_map, queries, B, d, kCM);
  if (s == HTAM_OK) s = make_bf16_tile_map(&hi_map, hi, G, d, kPageRows);
  if (s == HTAM_OK) s = make_bf16_tile_map(&lo_map, lo, G, d, kPageRows);
  if (s != HTAM_OK) return s;
  static std::atomic<uint64_t> attr_set{0};
  if (first_on_device(attr_set)) {
    HTAM_CK(cudaFuncSetAttribute(coarse_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCSmem));
  }
  const int nk = (int)ceil_div((int64_t)d, kCKBlock);
  const int kb_per = (int)ceil_div((int64_t)nk, splits);
  if (splits < 1 || (int)ceil_div((int64_t)nk, kb_per) != splits) return HTAM_EINVAL;  // no empty split
  dim3 grid((unsigned)ceil_div(B, kCM), (unsigned)ceil_div(G, kCN), (unsigned)splits);
  launch_kernel(coarse_tc_kernel, grid, kCThreads, kCSmem, st, q_map, hi_map, lo_map, d, kb_per, count, B, G, s1, status,
                                                     max_polls, gate);
  HTAM_CK_LAUNCH("coarse_tc_kernel");
  return HTAM_OK;
}

}  // namespace htam
