// fine_tc.cu -- fine scores on the tcgen05 tensor cores with a fused
// softmax-statistics and top-k epilogue.
//
// A work unit is (group g, chunk of up to 128 of the queries that selected g,
// segment of g's pages).  For each tile of 256 entries (two 128-row pages) the
// kernel computes S = Q_chunk (128 x D) * E_tile^T (D x 256) on the tensor
// cores: TMA stages 64-column K slices of both operands in shared memory with
// the 128-byte swizzle, one thread issues tcgen05.mma (M=128, N=256, K=16)
// into one of two fp32 accumulators in tensor memory, and four epilogue warps
// read the other accumulator back (tcgen05.ld, 32 columns at a time) while the
// next tile is being multiplied.  Each epilogue thread owns one query row:
//   * the online softmax statistics of s/tau over the unit's entries (the
//     Eq. 11 normaliser restricted by Eq. 12 to the selected groups), in the
//     log2 domain with ex2.approx;
//   * the row's K best (score, column) pairs so far, sorted, in registers
//     (the Eq. 13 pick as a top-k, K = k_entries rounded up to 8/16/32).
//     Scores that reach the admission bound are inserted one at a time
//     through an unrolled compare-and-swap pass over the list.  The bound
//     is the list's k-th score, raised by a per-query value that all units
//     of the query share through atomicMax after every tile: an entry below
//     it cannot reach the final top-k, since k other candidates score at
//     least as much.
// Columns are numbered in slot order within the unit, which is entry-id
// order within a group, so ties resolve to the lower entry id as everywhere
// else.  At the end of a unit each row writes one partial record (max, sum
// of exp, its top-k entry ids and scores) that the merge kernel combines.
//
// Units are taken dynamically (unit i by CTA i first, then from a global
// counter), so neighbouring units run at the same time -- the CTAs on the
// chunks of a large group read its pages at about the same moment -- and a
// CTA that drew short units takes more.  The producer warp takes each unit
// and passes its index to the MMA and epilogue warps through a small
// shared-memory queue guarded by mbarriers.
//
// Warp roles (192 threads, one CTA per SM, persistent over units):
//   warp 0   TMA producer (lane 0 issues)
//   warp 1   TMEM owner, MMA issuer (lane 0 issues)
//   warps 2..5  epilogue (TMEM lane quadrant = warp % 4)
// Every mbarrier wait is bounded; a give-up sets the memory's status word and
// the CTA drains its own copies and MMAs before releasing tensor memory.

#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "fine_tc.h"
#include "sm100.cuh"

namespace htam {

namespace {

using namespace sm100;

constexpr int kStages = 4;
constexpr int kKBlock = 64;                        // bf16 elements per 128-byte row slice
constexpr int kTileN = 2 * kPageRows;              // entries per tile (MMA N)
constexpr int kABytes = kTcRows * kKBlock * 2;     // 16 KiB
constexpr int kBBytes = kTileN * kKBlock * 2;      // 32 KiB
constexpr int kHalfB = kBBytes / 2;
constexpr int kThreads = 192;
constexpr uint32_t kAccCols = 256;                 // fp32 columns per accumulator
constexpr unsigned kFull = 0xffffffffu;

constexpr int kUQ = 4;  // unit queue slots (producer -> MMA and epilogue warps)

struct __align__(8) TcSmem {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  uint64_t uq_full[kUQ];   // a unit index was written
  uint64_t uq_empty[kUQ];  // the MMA warp and the 4 epilogue warps have read it
  uint32_t tmem_base;
  int abort;
  int uq[kUQ];             // unit indices in the order the producer took them; -1 = no more
};

// The j-th unit of this CTA, from the producer's queue, for a whole warp:
// -1 when there are no more units, or when the wait gave up (ok cleared).
__device__ __forceinline__ int take_unit(TcSmem *sh, int j, volatile int *abort, uint32_t max_polls, bool &ok) {
  const int slot = j % kUQ;
  if (!mbar_wait(&sh->uq_full[slot], (uint32_t)(j / kUQ) & 1u, abort, max_polls)) {
    ok = false;
    return -1;
  }
  const int u = *reinterpret_cast<volatile int *>(&sh->uq[slot]);
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&sh->uq_empty[slot]);
  return u;
}

constexpr size_t kSmemBytes = 1024 /* alignment slack */ + kStages * (kABytes + kBBytes) + sizeof(TcSmem);

__device__ __forceinline__ unsigned enc_score(float f) {
  unsigned u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float dec_score(unsigned u) {
  if (u == 0u) return -INFINITY;
  return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}

// A row's K best (score, column) pairs, best first, in registers.
template <int K>
struct RowTopK {
  float s[K];
  int c[K];

  __device__ __forceinline__ void init() {
#pragma unroll
    for (int i = 0; i < K; ++i) {
      s[i] = -INFINITY;
      c[i] = INT_MAX;
    }
  }

  // Inserts one pair whose column is above every column in the list (the
  // epilogue visits columns in increasing order), so on equal scores the
  // pair already in the list wins, which is the lower-column (lower-id) rule;
  // the worst pair falls off the end.  The list is sorted, so "slot i stays
  // ahead of x" holds for a prefix of the slots: slot i keeps its pair, takes
  // x, or takes slot i-1's pair depending only on its own and its
  // neighbour's comparison -- no dependency chain through the list.
  __device__ __forceinline__ void insert_later(float xs, int xc) {
    bool keep[K];
#pragma unroll
    for (int i = 0; i < K; ++i) keep[i] = s[i] >= xs;
#pragma unroll
    for (int i = K - 1; i >= 1; --i) {
      s[i] = keep[i] ? s[i] : (keep[i - 1] ? xs : s[i - 1]);
      c[i] = keep[i] ? c[i] : (keep[i - 1] ? xc : c[i - 1]);
    }
    s[0] = keep[0] ? s[0] : xs;
    c[0] = keep[0] ? c[0] : xc;
  }

  // The score at position k-1 (k <= K): the list is sorted, so it is the
  // smallest of the first k (a form that keeps the list in registers).
  __device__ __forceinline__ float kth(int k) const {
    float v = INFINITY;
#pragma unroll
    for (int i = 0; i < K; ++i) v = (i < k) ? fminf(v, s[i]) : v;
    return v;
  }
};

template <int K>
__global__ void __launch_bounds__(kThreads, 1)
    fine_tc_kernel(const __grid_constant__ CUtensorMap q_map, const __grid_constant__ CUtensorMap pool_map,
                   TcFineArgs a) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t *smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
  uint8_t *st_a = smem;
  uint8_t *st_b = st_a + kStages * kABytes;
  TcSmem *sh = reinterpret_cast<TcSmem *>(st_b + kStages * kBBytes);
  volatile int *abort = &sh->abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh->full[s], 1);
      mbar_init(&sh->empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh->acc_full[i], 1);
      mbar_init(&sh->acc_empty[i], 4);
    }
    mbar_init(&sh->drain, 1);
    for (int i = 0; i < kUQ; ++i) {
      mbar_init(&sh->uq_full[i], 1);
      mbar_init(&sh->uq_empty[i], 5);
    }
    sh->abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&q_map);
    prefetch_tensormap(&pool_map);
  }
  if (warp == 1) tmem_alloc(&sh->tmem_base, 2 * kAccCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = sh->tmem_base;
  const int n_units = *a.n_units;
  const int nk = (a.d + kKBlock - 1) / kKBlock;
  const int seg_pages = *a.seg_pages;

  // The producer and MMA warps run their loops with all 32 lanes (so every
  // warp reaches the final barrier converged); lane 0 issues the copies and
  // the MMAs.
  if (warp == 0) {
    // ---------------------------------------------------------- producer
    int st = 0;
    uint32_t ph = 0;
    uint32_t issued = 0, issued_phase = 0;  // per stage: a copy was issued / its phase parity
    bool ok = true;
    // Units are taken dynamically: unit blockIdx.x first, then the next one
    // from a global counter, so CTAs that drew short units take more.  Each
    // index goes through the queue to the MMA and epilogue warps.
    int u = blockIdx.x;
    for (int j = 0; ok; ++j) {
      const int slot = j % kUQ;
      if (!mbar_wait(&sh->uq_empty[slot], ((uint32_t)(j / kUQ) & 1u) ^ 1u, abort, a.max_polls)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        sh->uq[slot] = u < n_units ? u : -1;
        mbar_arrive(&sh->uq_full[slot]);
      }
      __syncwarp();
      if (u >= n_units) break;
      const int4 U = a.units[u];
      const int g = U.x;
      const int a_row = (a.q_direct ? 0 : a.bucket_off[g]) + U.y * kTcRows;
      const int pg0 = a.page_off[g];
      const int npg = a.page_off[g + 1] - pg0;
      const int p_beg = U.z * seg_pages, p_end = min(npg, p_beg + seg_pages);
      for (int p = p_beg; ok && p < p_end; p += 2) {
        const bool two = p + 1 < p_end;
        const int y0 = a.page_list[pg0 + p] * kPageRows;
        const int y1 = two ? a.page_list[pg0 + p + 1] * kPageRows : 0;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&sh->empty[st], ph ^ 1u, abort, a.max_polls)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            mbar_arrive_expect_tx(&sh->full[st], kABytes + (two ? kBBytes : kHalfB));
            const int x = kb * kKBlock;
            tma_load_2d(smem_addr(st_a + st * kABytes), &q_map, x, a_row, &sh->full[st]);
            tma_load_2d(smem_addr(st_b + st * kBBytes), &pool_map, x, y0, &sh->full[st]);
            if (two) tma_load_2d(smem_addr(st_b + st * kBBytes + kHalfB), &pool_map, x, y1, &sh->full[st]);
          }
          __syncwarp();
          issued |= 1u << st;
          issued_phase = (issued_phase & ~(1u << st)) | (ph << st);
          if (++st == kStages) {
            st = 0;
            ph ^= 1u;
          }
        }
      }
      int next = 0;
      if (lane == 0) next = (int)gridDim.x + atomicAdd(a.unit_ctr, 1);
      u = __shfl_sync(kFull, next, 0);
    }
    if (!ok && lane == 0) {
      atomicOr(a.status, 1u);
      sh->abort = 1;
    }
    // Drain: every copy issued has landed before the CTA exits.
    for (int s = 0; s < kStages; ++s) {
      if ((issued >> s) & 1u) {
        for (uint32_t i = 0; i < a.max_polls && !mbar_try_wait(&sh->full[s], (issued_phase >> s) & 1u); ++i) {
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // --------------------------------------------------------- MMA issuer
    const uint32_t idesc = idesc_bf16_f32(kTcRows, kTileN);
    int st = 0, acc = 0;
    uint32_t ph = 0, aph = 0;
    bool ok = true;
    for (int j = 0; ok; ++j) {
      const int u = take_unit(sh, j, abort, a.max_polls, ok);
      if (u < 0) break;
      const int4 U = a.units[u];
      const int g = U.x;
      const int npg = a.page_off[g + 1] - a.page_off[g];
      const int p_beg = U.z * seg_pages, p_end = min(npg, p_beg + seg_pages);
      for (int p = p_beg; ok && p < p_end; p += 2) {
        if (!mbar_wait(&sh->acc_empty[acc], aph ^ 1u, abort, a.max_polls)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tbase + acc * kAccCols;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&sh->full[st], ph, abort, a.max_polls)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0) {
            const uint64_t ad = sw128_kmajor_desc(smem_addr(st_a + st * kABytes));
            const uint64_t bd = sw128_kmajor_desc(smem_addr(st_b + st * kBBytes));
#pragma unroll
            for (int k = 0; k < kKBlock / 16; ++k) {
              umma_bf16(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kb | k) != 0);
            }
            umma_commit(&sh->empty[st]);
          }
          __syncwarp();
          if (++st == kStages) {
            st = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        if (lane == 0) umma_commit(&sh->acc_full[acc]);
        __syncwarp();
        if (++acc == 2) {
          acc = 0;
          aph ^= 1u;
        }
      }
    }
    if (!ok && lane == 0) {
      atomicOr(a.status, 1u);
      sh->abort = 1;
    }
    // Drain: all MMAs issued have completed.
    if (lane == 0) {
      umma_commit(&sh->drain);
      for (uint32_t i = 0; i < a.max_polls && !mbar_try_wait(&sh->drain, 0); ++i) {
      }
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------- epilogue
    const int quad = warp & 3;                // TMEM lane quadrant
    const int e = quad * 32 + lane;           // this thread's row of the chunk
    const uint32_t lane_addr = tbase + (static_cast<uint32_t>(quad * 32) << 16);
    const int k = a.ke;
    int acc = 0;
    uint32_t aph = 0;
    bool ok = true;
    RowTopK<K> top;
    for (int j = 0; ok; ++j) {
      const int u = take_unit(sh, j, abort, a.max_polls, ok);
      if (u < 0) break;
      const int4 U = a.units[u];
      const int g = U.x, c = U.y, sg = U.z;
      const int cg = a.cnt[g];
      const int nq = min(kTcRows, cg - c * kTcRows);
      const bool valid = e < nq;
      const int b = valid ? a.bucket[a.bucket_off[g] + c * kTcRows + e] : 0;
      float thr = valid ? dec_score(a.thr_enc[b]) : INFINITY;
      float m2 = -INFINITY, l = 0.f;
      top.init();
      const int pg0 = a.page_off[g];
      const int npg = a.page_off[g + 1] - pg0;
      const int cnt_rows = a.count[g];
      const int p_beg = sg * seg_pages, p_end = min(npg, p_beg + seg_pages);
      for (int p = p_beg; ok && p < p_end; p += 2) {
        const int f0 = min(kPageRows, cnt_rows - p * kPageRows);
        const int f1 = p + 1 < p_end ? min(kPageRows, cnt_rows - (p + 1) * kPageRows) : 0;
        if (valid) thr = fmaxf(thr, dec_score(a.thr_enc[b]));  // bounds published by other units
        if (!mbar_wait(&sh->acc_full[acc], aph, abort, a.max_polls)) ok = false;
        tc_fence_after();
        if (ok) {
#pragma unroll 1
          for (int ch = 0; ch < kTileN / 32; ++ch) {
            const int col0 = ch * 32;
            const int fill = ch < 4 ? f0 - col0 : f1 - (col0 - kPageRows);
            if (fill <= 0) continue;  // uniform across the warp
            uint32_t r[32];
            __syncwarp();             // converged for the warp-collective load
            tmem_ld32(lane_addr + acc * kAccCols + col0, r);
            tmem_wait_ld();
            const int nv = min(32, fill);
            const int cbase = (p - p_beg) * kPageRows + col0;  // unit column of r[0]
            uint32_t flagged = 0;
            if (valid) {
              float cmax = -INFINITY;
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (j < nv) cmax = fmaxf(cmax, __uint_as_float(r[j]));
              const float mz = cmax * a.k2;
              if (mz > m2) {
                l *= ex2(m2 - mz);
                m2 = mz;
              }
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                if (j < nv) {
                  const float s = __uint_as_float(r[j]);
                  l += ex2(fmaf(s, a.k2, -m2));
                  if (s >= thr) flagged |= 1u << j;
                }
              }
            }
            int most = __popc(flagged);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) most = max(most, __shfl_xor_sync(kFull, most, o));
            // Insert the flagged pairs one at a time.  (A sorting network over
            // the chunk costs more here: its unrolled code is large and runs
            // rarely, while this loop body is small.)
            for (int it = 0; it < most; ++it) {
              const bool any = flagged != 0u;
              const int j = any ? __ffs(flagged) - 1 : 0;
              flagged &= flagged - 1;
              // r[j] through a 5-level select tree on the bits of j.
              uint32_t t16[16], t8[8], t4[4], t2[2];
#pragma unroll
              for (int i = 0; i < 16; ++i) t16[i] = (j & 1) ? r[2 * i + 1] : r[2 * i];
#pragma unroll
              for (int i = 0; i < 8; ++i) t8[i] = (j & 2) ? t16[2 * i + 1] : t16[2 * i];
#pragma unroll
              for (int i = 0; i < 4; ++i) t4[i] = (j & 4) ? t8[2 * i + 1] : t8[2 * i];
#pragma unroll
              for (int i = 0; i < 2; ++i) t2[i] = (j & 8) ? t4[2 * i + 1] : t4[2 * i];
              const uint32_t xv = (j & 16) ? t2[1] : t2[0];
              if (any) top.insert_later(__uint_as_float(xv), cbase + j);
            }
            if (valid && most > 0) thr = fmaxf(thr, top.kth(k));
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->acc_empty[acc]);
        if (++acc == 2) {
          acc = 0;
          aph ^= 1u;
        }
        // Share this row's bound with the query's other units.
        if (valid && thr != -INFINITY && top.kth(k) == thr) atomicMax(&a.thr_enc[b], enc_score(thr));
      }
      if (!ok) break;
      if (valid) {
        const int64_t pidx = a.part_off[g] + (int64_t)sg * cg + c * kTcRows + e;
        a.part_ml[pidx] = make_float2(m2 * 0.69314718055994531f, l);
        // Unit columns -> entry ids: all page lookups, then all id loads,
        // then the stores, so the loads of a row overlap.
        int idv[K];
#pragma unroll
        for (int i = 0; i < K; ++i) {
          idv[i] = i < k && top.c[i] != INT_MAX ? a.page_list[pg0 + p_beg + top.c[i] / kPageRows] : -1;
        }
#pragma unroll
        for (int i = 0; i < K; ++i) {
          idv[i] = idv[i] >= 0 ? a.slot_id[(int64_t)idv[i] * kPageRows + top.c[i] % kPageRows] : INT_MAX;
        }
#pragma unroll
        for (int i = 0; i < K; ++i) {
          if (i < k) {
            a.part_s[pidx * k + i] = top.s[i];
            a.part_id[pidx * k + i] = idv[i];
          }
        }
      }
    }
    if (!ok && e == 0) {
      atomicOr(a.status, 1u);
      sh->abort = 1;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tbase, 2 * kAccCols);
  }
}

// Copies the query rows of tensor-core buckets into bucket order.
__global__ void gather_queries_kernel(const uint4 *__restrict__ Q, int vec_per_row, const int32_t *__restrict__ bucket,
                                      const int32_t *__restrict__ bucket_group, const int32_t *__restrict__ cnt,
                                      int tc_min, const int32_t *__restrict__ total_rows, int64_t max_rows,
                                      uint4 *__restrict__ Qg) {
  const int64_t r = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (r >= max_rows || r >= *total_rows) return;
  if (cnt[bucket_group[r]] < tc_min) return;
  const uint4 *src = Q + (int64_t)bucket[r] * vec_per_row;
  uint4 *dst = Qg + r * vec_per_row;
  for (int v = lane; v < vec_per_row; v += 32) dst[v] = src[v];
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess) {
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    } else {
      cudaGetLastError();
    }
  }
  return fn;
}

template <int K>
htam_status launch_k(const TcFineArgs &a, const CUtensorMap &q_map, const CUtensorMap &pool_map, int grid,
                     cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    HTAM_CK(cudaFuncSetAttribute(fine_tc_kernel<K>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes));
    attr_set = true;
  }
  fine_tc_kernel<K><<<grid, kThreads, kSmemBytes, st>>>(q_map, pool_map, a);
  HTAM_CK_LAUNCH("fine_tc_kernel");
  return HTAM_OK;
}

}  // namespace

htam_status make_bf16_tile_map(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto enc = encode_fn();
  if (!enc) return HTAM_ECUDA;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kKBlock), box_rows};
  cuuint32_t elem_strides[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
                   elem_strides, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? HTAM_OK : HTAM_ECUDA;
}

htam_status launch_gather_queries(const void *Q, int d, const int32_t *bucket, const int32_t *bucket_group,
                                  const int32_t *cnt, int tc_min, const int32_t *total_rows, int64_t max_rows,
                                  void *Qg, cudaStream_t st) {
  if (max_rows <= 0) return HTAM_OK;
  const int vec = d * 2 / 16;
  gather_queries_kernel<<<(unsigned)ceil_div(max_rows * 32, 256), 256, 0, st>>>(
      static_cast<const uint4 *>(Q), vec, bucket, bucket_group, cnt, tc_min, total_rows, max_rows,
      static_cast<uint4 *>(Qg));
  HTAM_CK_LAUNCH("gather_queries_kernel");
  return HTAM_OK;
}

htam_status launch_fine_tc(const TcFineArgs &a, const CUtensorMap &q_map, const CUtensorMap &pool_map, int grid,
                           cudaStream_t st) {
  if (grid <= 0) return HTAM_OK;
  if (a.ke <= 8) return launch_k<8>(a, q_map, pool_map, grid, st);
  if (a.ke <= 16) return launch_k<16>(a, q_map, pool_map, grid, st);
  return launch_k<32>(a, q_map, pool_map, grid, st);
}

}  // namespace htam
