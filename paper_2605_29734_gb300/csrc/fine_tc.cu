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
// Warp roles (224 threads, one CTA per SM, persistent over units):
//   warp 0   TMA producer (lane 0 issues)
//   warp 1   TMEM owner, MMA issuer (lane 0 issues)
//   warps 2..5  epilogue (TMEM lane quadrant = warp % 4)
//   warp 6   A copier: the chunk's query rows, straight from the query
//            matrix with cp.async into the swizzled A stages, two stages
//            ahead of their release (one-SM units of batches it is chosen
//            for; otherwise the block has 192 threads and the producer loads
//            bucket-ordered A tiles by TMA)
// Every mbarrier wait is bounded; a give-up sets the memory's status word and
// the CTA drains its own copies and MMAs before releasing tensor memory.

#include <cudaTypedefs.h>

#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "fine_tc.h"
#include "sm100.cuh"

namespace htam {

namespace {

using namespace sm100;

constexpr int kKBlock = 64;                        // bf16 elements per 128-byte row slice
constexpr int kTileN = 2 * kPageRows;              // entries per tile (MMA N)
constexpr int kABytes = kTcRows * kKBlock * 2;     // 16 KiB
constexpr int kBBytes = kTileN * kKBlock * 2;      // 32 KiB
constexpr int kHalfB = kBBytes / 2;                // one page's K slice
constexpr int kThreads = 224;     // with the A copier (warp 6)
constexpr int kThreadsTma = 192;  // without it: the A tiles come by TMA
constexpr int kALag = 2;  // stages the A copier keeps in flight before releasing the oldest
constexpr uint32_t kAccCols = 256;                 // fp32 columns per accumulator
constexpr unsigned kFull = 0xffffffffu;

// Operand ring per CTA: a single CTA stages A and both pages of B per K
// slice (48 KiB, 4 stages); a CTA of a pair stages A and its own page
// (32 KiB, 6 stages).
template <bool PAIR>
struct Ring {
  static constexpr int kStages = PAIR ? 6 : 4;
  static constexpr int kBStage = PAIR ? kHalfB : kBBytes;
};
constexpr int kMaxStages = 6;

constexpr int kUQ = 4;  // unit queue slots (producer -> MMA and epilogue warps)

struct __align__(8) TcSmem {
  uint64_t full[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  uint64_t uq_full[kUQ];   // a unit index was written
  uint64_t uq_empty[kUQ];  // every consumer of the slot has read it
  uint32_t tmem_base;
  int abort;
  int uq[kUQ];             // unit indices in the order the producer took them; -1 = no more
};

// The j-th unit of this CTA, from the producer's queue, for a whole warp:
// -1 when there are no more units, or when the wait gave up (ok cleared).
// Lane 0 then arrives on the slot's empty barrier, given by its
// shared::cluster address (rank 0's barrier for a CTA pair).
template <bool PAIR>
__device__ __forceinline__ int take_unit(TcSmem *sh, int j, uint32_t empty_caddr0, volatile int *abort,
                                         uint32_t max_polls, bool &ok) {
  const int slot = j % kUQ;
  const uint32_t par = (uint32_t)(j / kUQ) & 1u;
  if (!(PAIR ? mbar_wait_cluster(&sh->uq_full[slot], par, abort, max_polls)
             : mbar_wait(&sh->uq_full[slot], par, abort, max_polls))) {
    ok = false;
    return -1;
  }
  const int u = *reinterpret_cast<volatile int *>(&sh->uq[slot]);
  __syncwarp();
  if ((threadIdx.x & 31) == 0) {
    if constexpr (PAIR) {
      mbar_arrive_cluster(empty_caddr0 + slot * (uint32_t)sizeof(uint64_t));
    } else {
      mbar_arrive(&sh->uq_empty[slot]);
    }
  }
  return u;
}

// Copies of query rows into an A stage by the copier warp's lanes: 16 bytes
// each, zero-filled past the row's end (src_bytes 0).
__device__ __forceinline__ void cp_async16_zfill(uint32_t dst, const void *src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// Makes this thread's completed generic-proxy writes to shared memory (the
// copies above) visible to the async proxy that tcgen05.mma reads through.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Per epilogue warp, a 32 x 32 fp32 staging area: a lane writes its row's
// 32-column accumulator chunk there when some lane of the warp has pairs to
// insert, and reads back the flagged columns one at a time by index.
constexpr int kEpiWarps = 4;
constexpr int kStageFloats = 32 * 32;

template <bool PAIR>
constexpr size_t smem_bytes() {
  return 1024 /* alignment slack */ + Ring<PAIR>::kStages * (kABytes + Ring<PAIR>::kBStage) +
         sizeof(float) * kEpiWarps * kStageFloats + sizeof(TcSmem);
}

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

  // The score at position k-1 (1 <= k <= K) of the sorted list, through a
  // select tree on the bits of k-1 (log2 K levels instead of a K-long chain;
  // register indices stay static).
  __device__ __forceinline__ float kth(int k) const {
    if (k == K) return s[K - 1];
    const int i = k - 1;
    float t[K];
#pragma unroll
    for (int j = 0; j < K; ++j) t[j] = s[j];
#pragma unroll
    for (int w = K / 2, bit = 1; w >= 1; w /= 2, bit *= 2) {
#pragma unroll
      for (int j = 0; j < w; ++j) t[j] = (i & bit) ? t[2 * j + 1] : t[2 * j];
    }
    return t[0];
  }
};

// PAIR = false: one CTA per unit (group, 128-query chunk, page segment).
// PAIR = true: a cluster of two CTAs per unit (group, pair of chunks 2cp and
// 2cp+1, page segment), multiplying with tcgen05.mma.cta_group::2 (M=256:
// rank r holds chunk 2cp+r's 128 queries as its A rows and the tile's page r
// as its half of B, N=256).  Each CTA reads half of the entry bytes a single
// CTA reads per MMA, so its operand ring holds six K slices instead of four.
// Rank 0 takes the units and passes them to both CTAs' queues, sets the
// byte count each stage expects from both CTAs' copies, and issues the MMAs
// and their commits to the barriers of both CTAs; each rank's epilogue
// reads its own 128 accumulator rows.
template <int K, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1)
    fine_tc_kernel(const __grid_constant__ CUtensorMap q_map, const __grid_constant__ CUtensorMap pool_map,
                   TcFineArgs a) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  constexpr int kStages = Ring<PAIR>::kStages;
  constexpr int kBStage = Ring<PAIR>::kBStage;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t *smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
  uint8_t *st_a = smem;
  uint8_t *st_b = st_a + kStages * kABytes;
  float *st_epi = reinterpret_cast<float *>(st_b + kStages * kBStage);  // [kEpiWarps][32][32]
  TcSmem *sh = reinterpret_cast<TcSmem *>(st_epi + kEpiWarps * kStageFloats);
  volatile int *abort = &sh->abort;

  // No units (every bucket went to the CUDA cores): leave before setting up
  // (uniform over the grid, so a CTA pair leaves together).
  if (*a.n_units == 0) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  // Rank 0's barriers as shared::cluster addresses (this CTA's own when single).
  const uint32_t full_c0 = PAIR ? mapa_shared(smem_addr(&sh->full[0]), 0) : smem_addr(&sh->full[0]);
  const uint32_t acc_empty_c0 = PAIR ? mapa_shared(smem_addr(&sh->acc_empty[0]), 0) : smem_addr(&sh->acc_empty[0]);
  const uint32_t uq_empty_c0 = PAIR ? mapa_shared(smem_addr(&sh->uq_empty[0]), 0) : smem_addr(&sh->uq_empty[0]);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      // With the A copier, a stage is full once its B pages' bytes landed
      // and the copier has arrived for its A rows.
      mbar_init(&sh->full[s], (!PAIR && a.a_rows) ? 2 : 1);
      mbar_init(&sh->empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh->acc_full[i], 1);
      mbar_init(&sh->acc_empty[i], PAIR ? 8 : 4);  // the epilogue warps of every CTA of the unit
    }
    mbar_init(&sh->drain, 1);
    for (int i = 0; i < kUQ; ++i) {
      mbar_init(&sh->uq_full[i], 1);
      // Single: MMA warp + 4 epilogue warps (+ the A copier).  Pair (rank 0's
      // barrier): its MMA warp and 4 epilogue warps, rank 1's producer and 4
      // epilogue warps.
      mbar_init(&sh->uq_empty[i], PAIR ? 10 : (a.a_rows ? 6 : 5));
    }
    sh->abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&q_map);
    prefetch_tensormap(&pool_map);
  }
  if constexpr (PAIR) {
    cluster_sync();  // both CTAs' barriers are initialised before any remote arrival
    if (warp == 1) tmem_alloc_pair(&sh->tmem_base, 2 * kAccCols);
  } else {
    if (warp == 1) tmem_alloc(&sh->tmem_base, 2 * kAccCols);
  }
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
    // Units are taken dynamically: unit (cluster) index first, then the next
    // one from a global counter, so CTAs that drew short units take more.
    // Each index goes through the queue to the MMA and epilogue warps (of
    // both CTAs of a pair; rank 1's producer reads rank 0's choice).
    int u = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
    const int n_slots = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
    for (int j = 0; ok; ++j) {
      const int slot = j % kUQ;
      if (leader) {
        if (!mbar_wait(&sh->uq_empty[slot], ((uint32_t)(j / kUQ) & 1u) ^ 1u, abort, a.max_polls)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          const int v = u < n_units ? u : -1;
          sh->uq[slot] = v;
          mbar_arrive(&sh->uq_full[slot]);
          if constexpr (PAIR) {
            st_cluster_u32(mapa_shared(smem_addr(&sh->uq[slot]), 1), (uint32_t)v);
            mbar_arrive_cluster(mapa_shared(smem_addr(&sh->uq_full[slot]), 1));
          }
        }
        __syncwarp();
      } else {
        u = take_unit<PAIR>(sh, j, uq_empty_c0, abort, a.max_polls, ok);
        if (!ok) break;
        if (u < 0) u = n_units;
      }
      if (u >= n_units) break;
      const int4 U = a.units[u];
      const int g = U.x;
      // This CTA's chunk; a pair's missing second chunk re-reads the first
      // chunk's rows (its accumulator rows are never read).
      int c = U.y;
      if constexpr (PAIR) {
        c = 2 * U.y + (int)rank;
        if (c * kTcRows >= a.cnt[g]) c = 2 * U.y;
      }
      const int a_row = (a.q_direct ? 0 : a.bucket_off[g]) + c * kTcRows;
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
            const int x = kb * kKBlock;
            const uint32_t dst_a = smem_addr(st_a + st * kABytes), dst_b = smem_addr(st_b + st * kBStage);
            if constexpr (PAIR) {
              // Both CTAs' copies complete on rank 0's barrier; rank 0
              // expects both ranks' A rows and the tile's pages.
              const uint32_t bar = full_c0 + st * (uint32_t)sizeof(uint64_t);
              if (leader) mbar_arrive_expect_tx(&sh->full[st], 2 * kABytes + (two ? 2 * kHalfB : kHalfB));
              tma_load_2d_pair(dst_a, &q_map, x, a_row, bar);
              if (leader) {
                tma_load_2d_pair(dst_b, &pool_map, x, y0, bar);
              } else if (two) {
                tma_load_2d_pair(dst_b, &pool_map, x, y1, bar);
              }
            } else if (a.a_rows) {
              mbar_arrive_expect_tx(&sh->full[st], two ? kBBytes : kHalfB);
              tma_load_2d(dst_b, &pool_map, x, y0, &sh->full[st]);
              if (two) tma_load_2d(dst_b + kHalfB, &pool_map, x, y1, &sh->full[st]);
            } else {
              mbar_arrive_expect_tx(&sh->full[st], kABytes + (two ? kBBytes : kHalfB));
              tma_load_2d(dst_a, &q_map, x, a_row, &sh->full[st]);
              tma_load_2d(dst_b, &pool_map, x, y0, &sh->full[st]);
              if (two) tma_load_2d(dst_b + kHalfB, &pool_map, x, y1, &sh->full[st]);
            }
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
      if (leader) {
        int next = 0;
        if (lane == 0) next = n_slots + atomicAdd(a.unit_ctr, 1);
        u = __shfl_sync(kFull, next, 0);
      }
    }
    if (!ok && lane == 0) {
      atomicOr(a.status, 1u);
      sh->abort = 1;
    }
    // Drain: every copy issued has landed before the CTA exits.  A single
    // CTA (and rank 0) polls the stage's full barrier; rank 1's copies
    // complete on rank 0's barrier, so rank 1 polls its empty barrier, which
    // the MMAs release only after both CTAs' copies of the stage landed.
    for (int s = 0; s < kStages; ++s) {
      if ((issued >> s) & 1u) {
        const uint32_t par = (issued_phase >> s) & 1u;
        uint64_t *bar = leader ? &sh->full[s] : &sh->empty[s];
        for (uint32_t i = 0; i < a.max_polls && !mbar_try_wait(bar, par); ++i) {
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // --------------------------------------------------------- MMA issuer
    // (rank 0 of a pair issues for both CTAs; rank 1's MMA warp only holds
    // its share of the tensor memory allocation)
    const uint32_t idesc = idesc_bf16_f32(PAIR ? 2 * kTcRows : kTcRows, kTileN);
    int st = 0, acc = 0;
    uint32_t ph = 0, aph = 0;
    bool ok = true;
    for (int j = 0; ok && leader; ++j) {
      const int u = take_unit<PAIR>(sh, j, uq_empty_c0, abort, a.max_polls, ok);
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
            const uint64_t bd = sw128_kmajor_desc(smem_addr(st_b + st * kBStage));
#pragma unroll
            for (int k = 0; k < kKBlock / 16; ++k) {
              if constexpr (PAIR) {
                umma_bf16_pair(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kb | k) != 0);
              } else {
                umma_bf16(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kb | k) != 0);
              }
            }
            if constexpr (PAIR) {
              umma_commit_pair(&sh->empty[st], 0x3);
            } else {
              umma_commit(&sh->empty[st]);
            }
          }
          __syncwarp();
          if (++st == kStages) {
            st = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        if (lane == 0) {
          if constexpr (PAIR) {
            umma_commit_pair(&sh->acc_full[acc], 0x3);
          } else {
            umma_commit(&sh->acc_full[acc]);
          }
        }
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
    if (leader && lane == 0) {
      if constexpr (PAIR) {
        umma_commit_pair(&sh->drain, 0x1);
      } else {
        umma_commit(&sh->drain);
      }
      for (uint32_t i = 0; i < a.max_polls && !mbar_try_wait(&sh->drain, 0); ++i) {
      }
    }
    __syncwarp();
  } else if (warp == 6) {
    // ---------------------------------------------------------- A copier
    // Walks the same units, tiles and K slices as the producer (so the
    // same stages and phases), waits for each stage to be free, copies the
    // K slice of the chunk's 128 query rows into it, and releases a stage
    // kALag stages later: once the lane's copy group of that stage
    // completed, a proxy fence, then one arrival.  Lane l holds the query
    // ids of rows l, l+32, l+64 and l+96.
    if (!PAIR && a.a_rows) {
      int st = 0;
      uint32_t ph = 0;
      bool ok = true;
      int64_t n_iss = 0;  // stages issued (their stage indices run in order)
      int qid[4];         // query ids of the chunk's rows lane, lane+32, lane+64, lane+96
      for (int j = 0; ok; ++j) {
        const int u = take_unit<PAIR>(sh, j, uq_empty_c0, abort, a.max_polls, ok);
        if (u < 0) break;
        const int4 U = a.units[u];
        const int g = U.x, c = U.y;
        const int a_row = a.bucket_off[g] + c * kTcRows;
        const int nq = min(kTcRows, a.cnt[g] - c * kTcRows);
        // Rows past the chunk's queries repeat its first query (in bounds;
        // their accumulator rows are never read).
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int r = lane + 32 * i;
          qid[i] = a.bucket[a_row + (r < nq ? r : 0)];
        }
        const int npg = a.page_off[g + 1] - a.page_off[g];
        const int p_beg = U.z * seg_pages, p_end = min(npg, p_beg + seg_pages);
        const int n_stages = (p_end - p_beg + 1) / 2 * nk;
        for (int i_st = 0; i_st < n_stages; ++i_st) {
          const int kb = i_st % nk;
          if (!mbar_wait(&sh->empty[st], ph ^ 1u, abort, a.max_polls)) {
            ok = false;
            break;
          }
          // K slice kb of the 128 rows, four rows per instruction: eight lanes
          // take the eight 16-byte vectors of one row (128 contiguous bytes),
          // stored where the 128-byte swizzle puts them (vector v of row r at
          // 16 * (v ^ (r % 8))).  The row's query id comes from the lane that
          // holds it.
          const uint32_t dst_a = smem_addr(st_a + st * kABytes);
          const int v = lane & 7;
          const bool in = kb * (kKBlock / 8) + v < a.qvec;
          const int vsrc = in ? kb * (kKBlock / 8) + v : 0;
#pragma unroll
          for (int i = 0; i < kTcRows / 4; ++i) {
            const int r = 4 * i + (lane >> 3);
            const int q = __shfl_sync(kFull, qid[i / 8], r & 31);
            cp_async16_zfill(dst_a + r * 128 + ((v ^ (r & 7)) << 4), a.queries + (int64_t)q * a.qvec + vsrc,
                             in ? 16u : 0u);
          }
          cp_async_commit();
          if (++n_iss > kALag) {
            // The stage issued kALag stages ago: its group has completed.
            cp_async_wait<kALag>();
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh->full[(st + kStages - kALag) % kStages]);
          }
          if (++st == kStages) {
            st = 0;
            ph ^= 1u;
          }
        }
      }
      // The stages still waiting: every copy of the lane completed, fenced,
      // then their arrivals.
      cp_async_wait<0>();
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int left = (int)(n_iss < kALag ? n_iss : kALag);
        for (int q = left; q >= 1; --q) mbar_arrive(&sh->full[(st + kStages - q) % kStages]);
      }
      if (!ok && lane == 0) {
        atomicOr(a.status, 1u);
        sh->abort = 1;
      }
    }
  } else {
    // ----------------------------------------------------------- epilogue
    const int quad = warp & 3;                // TMEM lane quadrant
    const int e = quad * 32 + lane;           // this thread's row of the chunk
    const uint32_t lane_addr = tbase + (static_cast<uint32_t>(quad * 32) << 16);
    const int k = a.ke;
    const int kj = (k + kThrSlots - 1) / kThrSlots;  // the rank each segment class publishes
    // This lane's staging row (16-byte groups swizzled by the lane so that
    // the warp's row writes spread over the banks).
    float *stg = st_epi + (warp - 2) * kStageFloats + lane * 32;
    int acc = 0;
    uint32_t aph = 0;
    bool ok = true;
    RowTopK<K> top;
    for (int j = 0; ok; ++j) {
      const int u = take_unit<PAIR>(sh, j, uq_empty_c0, abort, a.max_polls, ok);
      if (u < 0) break;
      const int4 U = a.units[u];
      const int g = U.x, sg = U.z;
      const int c = PAIR ? 2 * U.y + (int)rank : U.y;
      const int cg = a.cnt[g];
      const int nq = min(kTcRows, cg - c * kTcRows);  // <= 0: a pair's missing second chunk
      const bool valid = e < nq;
      const int b = valid ? a.bucket[a.bucket_off[g] + c * kTcRows + e] : 0;
      unsigned *tb = a.thr_enc + (int64_t)b * kThrWords;
      const int cls = 1 + sg % kThrSlots;
      float thr = valid ? -INFINITY : INFINITY;
      // The query's shared bounds, read one tile ahead: the loads' latency
      // is spent in the previous tile's work instead of stalling this one.
      // (L2 loads: other CTAs raise the words with atomics.)
      unsigned w0 = 0u, w1 = 0u, w2 = 0u, w3 = 0u, w4 = 0u;
      auto load_bounds = [&]() {
        w0 = __ldcg(tb);
        w1 = __ldcg(tb + 1);
        w2 = __ldcg(tb + 2);
        w3 = __ldcg(tb + 3);
        w4 = __ldcg(tb + 4);
      };
      auto shared_bound = [&]() {
        const float slots = fminf(fminf(dec_score(w1), dec_score(w2)), fminf(dec_score(w3), dec_score(w4)));
        return fmaxf(dec_score(w0), slots);
      };
      if (valid) load_bounds();
      float pub_k = -INFINITY, pub_j = -INFINITY;  // what this unit has published
      float m2 = -INFINITY, l = 0.f;
      top.init();
      const int pg0 = a.page_off[g];
      const int npg = a.page_off[g + 1] - pg0;
      const int cnt_rows = a.count[g];
      const int p_beg = sg * seg_pages, p_end = min(npg, p_beg + seg_pages);
      for (int p = p_beg; ok && p < p_end; p += 2) {
        const int f0 = min(kPageRows, cnt_rows - p * kPageRows);
        const int f1 = p + 1 < p_end ? min(kPageRows, cnt_rows - (p + 1) * kPageRows) : 0;
        if (!mbar_wait(&sh->acc_full[acc], aph, abort, a.max_polls)) ok = false;
        tc_fence_after();
        if (ok && nq > 0) {
          // One 32-column chunk of the accumulator row: softmax statistics,
          // then the pairs that reach the bound into the row's top-k.
          auto chunk = [&](const uint32_t (&r)[32], int ch) {
            const int col0 = ch * 32;
            const int fill = ch < 4 ? f0 - col0 : f1 - (col0 - kPageRows);
            const int nv = min(32, fill);
            const int cbase = (p - p_beg) * kPageRows + col0;  // unit column of r[0]
            uint32_t flagged = 0;
            if (valid) {
              // With one epilogue warp per scheduler the chunk's arithmetic
              // is latency-bound, so it runs as short independent chains:
              // the maximum by a tree of three-input maxima, the sum of
              // exponentials in four interleaved partial sums, the flags
              // only on a lane whose maximum reaches its bound, built in
              // four partial masks.  A full chunk (every page row filled,
              // uniform across the warp) skips the per-column fill test.
              auto body = [&](auto full_tag) {
                constexpr bool kFullChunk = decltype(full_tag)::value;
                auto val = [&](int j) {
                  return (kFullChunk || j < nv) ? __uint_as_float(r[j]) : -INFINITY;
                };
                float t[11];
#pragma unroll
                for (int i = 0; i < 10; ++i) t[i] = max3f(val(3 * i), val(3 * i + 1), val(3 * i + 2));
                t[10] = fmaxf(val(30), val(31));
                const float cmax = max3f(max3f(t[0], t[1], t[2]), max3f(t[3], t[4], t[5]),
                                         max3f(max3f(t[6], t[7], t[8]), t[9], t[10]));
                const float mz = cmax * a.k2;
                if (mz > m2) {
                  l *= ex2(m2 - mz);
                  m2 = mz;
                }
                float l4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int j = 0; j < 32; ++j) l4[j & 3] += ex2(fmaf(val(j), a.k2, -m2));
                l += (l4[0] + l4[1]) + (l4[2] + l4[3]);
                if (cmax >= thr) {
                  uint32_t f4[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                  for (int j = 0; j < 32; ++j) {
                    if ((kFullChunk || j < nv) && val(j) >= thr) f4[j & 3] |= 1u << j;
                  }
                  flagged = (f4[0] | f4[1]) | (f4[2] | f4[3]);
                }
              };
              if (nv == 32) {
                body(std::true_type{});
              } else {
                body(std::false_type{});
              }
            }
            const int most = (int)__reduce_max_sync(kFull, (unsigned)__popc(flagged));
            // Insert the flagged pairs one at a time.  (A sorting network over
            // the chunk costs more here: its unrolled code is large and runs
            // rarely, while this loop body is small.)  The chunk goes through
            // this lane's staging row, so a flagged column is one indexed
            // load; each lane reads only what it wrote, so no barrier.
            if (most > 0) {
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                *reinterpret_cast<uint4 *>(stg + ((i ^ (lane & 7)) << 2)) =
                    make_uint4(r[4 * i], r[4 * i + 1], r[4 * i + 2], r[4 * i + 3]);
              }
            }
            for (int it = 0; it < most; ++it) {
              const bool any = flagged != 0u;
              const int j = any ? __ffs(flagged) - 1 : 0;
              flagged &= flagged - 1;
              const float xv = stg[(((j >> 2) ^ (lane & 7)) << 2) | (j & 3)];
              if (any) top.insert_later(xv, cbase + j);
            }
            if (valid && most > 0) thr = fmaxf(thr, top.kth(k));
          };
          // The chunks holding entries are a prefix (only a group's last page
          // is partly filled, and nothing follows it).  Each chunk's load is
          // issued before the previous chunk is processed, so the tensor
          // memory reads overlap the arithmetic.
          const int n_ch = f1 > 0 ? 4 + (f1 + 31) / 32 : (f0 + 31) / 32;
          const uint32_t acc_addr = lane_addr + acc * kAccCols;
          uint32_t ra[32], rb[32];
          __syncwarp();  // converged for the warp-collective loads and waits
          tmem_ld32(acc_addr, ra);
          tmem_wait_ld(ra);
          if (valid) thr = fmaxf(thr, shared_bound());  // bounds published by other units
#pragma unroll 1
          for (int ch = 0; ch < n_ch; ch += 2) {
            const bool has_b = ch + 1 < n_ch;  // uniform across the warp
            __syncwarp();
            if (has_b) tmem_ld32(acc_addr + (ch + 1) * 32, rb);
            chunk(ra, ch);
            __syncwarp();
            tmem_wait_ld(rb);
            if (!has_b) break;
            if (ch + 2 < n_ch) tmem_ld32(acc_addr + (ch + 2) * 32, ra);
            chunk(rb, ch + 1);
            __syncwarp();
            tmem_wait_ld(ra);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (PAIR) {
            mbar_arrive_cluster(acc_empty_c0 + acc * (uint32_t)sizeof(uint64_t));
          } else {
            mbar_arrive(&sh->acc_empty[acc]);
          }
        }
        if (++acc == 2) {
          acc = 0;
          aph ^= 1u;
        }
        // Share this row's bounds with the query's other units (its k-th
        // score, and its kj-th score in its segment class), and read theirs
        // for the next tile.
        if (valid) {
          const float kv = top.kth(k);
          if (kv > pub_k) {
            atomicMax(tb, enc_score(kv));
            pub_k = kv;
          }
          const float jv = top.kth(kj);
          if (jv > pub_j) {
            atomicMax(tb + cls, enc_score(jv));
            pub_j = jv;
          }
          load_bounds();
        }
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
  if constexpr (PAIR) {
    cluster_sync();  // rank 0's MMAs (which use both CTAs' memory) have drained
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc_pair(tbase, 2 * kAccCols);
    }
    cluster_sync();
  } else {
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tbase, 2 * kAccCols);
    }
  }
}

// Copies the query rows of tensor-core buckets into bucket order.
__global__ void gather_queries_kernel(const uint4 *__restrict__ Q, int vec_per_row, const int32_t *__restrict__ bucket,
                                      const int32_t *__restrict__ bucket_group, const int32_t *__restrict__ cnt,
                                      int tc_min, const int32_t *__restrict__ total_rows, int64_t max_rows,
                                      uint4 *__restrict__ Qg) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
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

template <int K, bool PAIR>
htam_status launch_k(const TcFineArgs &a, const CUtensorMap &q_map, const CUtensorMap &pool_map, int grid,
                     cudaStream_t st) {
  static std::atomic<uint64_t> attr_set{0};
  if (first_on_device(attr_set)) {
    HTAM_CK(cudaFuncSetAttribute(fine_tc_kernel<K, PAIR>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem_bytes<PAIR>()));
  }
  if constexpr (PAIR) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid, 1, 1);
    cfg.blockDim = dim3(kThreadsTma, 1, 1);
    cfg.dynamicSmemBytes = smem_bytes<PAIR>();
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_launch_pdl ? 2 : 1;
    HTAM_CK(cudaLaunchKernelEx(&cfg, fine_tc_kernel<K, true>, q_map, pool_map, a));
  } else {
    launch_kernel(fine_tc_kernel<K, false>, grid, a.a_rows ? kThreads : kThreadsTma, smem_bytes<false>(), st, q_map,
                  pool_map, a);
  }
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
  launch_kernel(gather_queries_kernel, (unsigned)ceil_div(max_rows * 32, 256), 256, 0, st, 
      static_cast<const uint4 *>(Q), vec, bucket, bucket_group, cnt, tc_min, total_rows, max_rows,
      static_cast<uint4 *>(Qg));
  HTAM_CK_LAUNCH("gather_queries_kernel");
  return HTAM_OK;
}

htam_status launch_fine_tc(const TcFineArgs &a, const CUtensorMap &q_map, const CUtensorMap &pool_map, int grid,
                           bool pair, cudaStream_t st) {
  if (pair) grid &= ~1;  // whole clusters
  if (grid <= 0) return HTAM_OK;
  if (pair) {
    if (a.ke <= 8) return launch_k<8, true>(a, q_map, pool_map, grid, st);
    if (a.ke <= 16) return launch_k<16, true>(a, q_map, pool_map, grid, st);
    return launch_k<32, true>(a, q_map, pool_map, grid, st);
  }
  if (a.ke <= 8) return launch_k<8, false>(a, q_map, pool_map, grid, st);
  if (a.ke <= 16) return launch_k<16, false>(a, q_map, pool_map, grid, st);
  return launch_k<32, false>(a, q_map, pool_map, grid, st);
}

}  // namespace htam
