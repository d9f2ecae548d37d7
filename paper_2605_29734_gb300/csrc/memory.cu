// memory.cu -- building and appending to the paged group memory.
//
// The memory mirrors the paper's Hierarchical Transition Graph (Eq. 6, §4.1):
// entries (local nodes) are filed under their parent group (global node), and
// each group keeps a key equal to the mean of its entries.  Appending is the
// memory update of Eq. 15: new rows go to the tail of their group's pages and
// the touched groups' keys are updated in place from fp64 running sums.
//
// Every step is deterministic: rows are placed by a stable counting sort (the
// i-th row of a group in input order lands at the group's next free slot), and
// key sums are taken over rows in slot order, in fixed-size row segments whose
// compensated fp32 partials are added to the fp64 sum in segment order.

#include <algorithm>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace htam {

namespace {

constexpr int kKeySegRowsMin = 16;     // rows per key partial-sum segment: at least this,
constexpr int kKeySegRowsMax = 1024;   // at most this,
constexpr int64_t kKeySegTarget = 4096;  // and about count / this (bounds the partial-sum buffer)

// Rows per key segment for a batch of `count` rows: short segments for
// appends (many blocks in parallel), long ones for large builds (a partial
// sum buffer of about kKeySegTarget + n_groups segments).
static int key_seg_rows(int64_t count) {
  int r = kKeySegRowsMin;
  while (r < kKeySegRowsMax && (int64_t)r * kKeySegTarget < count) r *= 2;
  return r;
}

// Per-group counts of a batch, and the stable sort's per (group, chunk of
// `chunk` rows) counts hist[g * n_chunks + c] (both zeroed before).  Ids of
// -1 (no group given) are counted apart when `allow_unassigned` (the
// nearest-key assignment adds them later), and count as bad otherwise; any
// other id outside [0, n_groups) sets `bad`.
__global__ void count_groups_kernel(const int32_t *__restrict__ gid, int64_t n, int32_t n_groups,
                                    int allow_unassigned, int32_t *__restrict__ counts, int32_t *__restrict__ bad,
                                    int32_t *__restrict__ unassigned, int32_t *__restrict__ hist, int64_t chunk,
                                    int64_t n_chunks) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n; e += stride) {
    int32_t g = gid[e];
    if (g == -1 && allow_unassigned) {
      atomicAdd(unassigned, 1);
    } else if (g < 0 || g >= n_groups) {
      atomicOr(bad, 1);
    } else {
      atomicAdd(&counts[g], 1);
      atomicAdd(&hist[(int64_t)g * n_chunks + e / chunk], 1);
    }
  }
}

// The group of row e: its given id, or for a row given -1 the group the
// nearest-key assignment chose.
__device__ __forceinline__ int32_t row_group(const int32_t *__restrict__ gid, const int32_t *__restrict__ ids,
                                             int64_t e) {
  const int32_t g = gid[e];
  return g >= 0 ? g : ids[e];
}

struct KeySeg {
  int32_t g, r0, r1, pad;
};
struct KeyGroup {
  int32_t g, seg0, seg1, count;
  double inv;  // 1 / count (0 for an empty group), taken once per group by the layout block
};

// Inclusive scan of one value per thread over a block of kLayoutThreads.
constexpr int kLayoutThreads = 1024;
__device__ __forceinline__ int64_t block_scan_incl(int64_t v, int64_t *sh /* [32] */) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t t = __shfl_up_sync(kFullMask, v, o);
    if (lane >= o) v += t;
  }
  if (lane == 31) sh[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int64_t w = lane < kLayoutThreads / 32 ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t t = __shfl_up_sync(kFullMask, w, o);
      if (lane >= o) w += t;
    }
    sh[lane] = w;
  }
  __syncthreads();
  const int64_t r = v + (warp > 0 ? sh[warp - 1] : 0);
  __syncthreads();  // sh is reused by the next scan
  return r;
}

// One block lays out a batch on the device (the page layout, the key
// segments, the new sizes), so an append needs no host round trip.
//   per group g: old = count[g], add = bcount[g], new = old + add;
//   pages: ceil(new/128) in total, of which the ones beyond ceil(old/128)
//     are fresh pages taken from the pool cursor dev_ctr[1] in group order;
//   page_off_new = the exclusive scan of the page totals; first_new[g] =
//     g's first fresh page;
//   key segments over the new rows of every touched group (rows old.. new in
//     steps of seg_rows) and one KeyGroup per touched group;
//   base[g] = old (the stable sort's starting slot), count[g] = new;
//   meta[0..1] = segment and touched-group counts, *id_base = the entry count
//     before the batch, and the entry count grows by `rows`.
// A bad batch changes nothing: the current offsets are copied to the new
// layout, no segment is listed, and status bit 1 records the rejection.
// For small batches and layouts the same block then does what
// group_lists_kernel does (the chunk scan when fuse_scan, the page list copy
// when fuse_copy).
__device__ void chunk_scan_group(int g, int lane, int32_t *hist, int64_t n_chunks, const int32_t *base);
__device__ void page_copy_group(int g, int lane, const int32_t *page_off_cur, const int32_t *page_list_cur,
                                const int32_t *page_off_new, const int32_t *first_new, int32_t *page_list_new);

__global__ void __launch_bounds__(kLayoutThreads, 1)
    layout_kernel(int32_t G, int64_t rows, int seg_rows, int32_t *__restrict__ bcount,
                  const int32_t *__restrict__ bad, int32_t *__restrict__ count,
                  const int32_t *__restrict__ page_off_cur, int32_t *__restrict__ page_off_new,
                  int32_t *__restrict__ first_new, int32_t *__restrict__ base, KeySeg *__restrict__ segs,
                  KeyGroup *__restrict__ kgroups, int32_t *__restrict__ meta, int64_t *__restrict__ id_base,
                  int64_t *__restrict__ dev_ctr, unsigned *__restrict__ status, int fuse_scan, int32_t *hist,
                  int64_t n_chunks, int fuse_copy, const int32_t *page_list_cur, int32_t *page_list_new) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  __shared__ int64_t sh[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (*bad) {  // uniform over the block
    for (int g = threadIdx.x; g <= G; g += blockDim.x) page_off_new[g] = page_off_cur[g];
    // The batch's group counts and its count of rows without a group are
    // read by nothing after this block: cleared here for the next batch.
    for (int g = threadIdx.x; g < G; g += blockDim.x) bcount[g] = 0;
    if (threadIdx.x == 0) {
      meta[0] = 0;
      meta[1] = 0;
      atomicOr(status, 2u);
      bcount[G + 1] = 0;
    }
    if (fuse_copy) {
      __syncthreads();
      for (int g = warp; g < G; g += kLayoutThreads / 32) {
        page_copy_group(g, lane, page_off_cur, page_list_cur, page_off_new, first_new, page_list_new);
      }
    }
    return;
  }
  const int per = (int)ceil_div(G, kLayoutThreads);
  const int g0 = min(G, (int)threadIdx.x * per), g1 = min(G, g0 + per);
  int64_t tp = 0, np = 0, ns = 0, nt = 0;  // this thread's pages, fresh pages, segments, touched groups
  for (int g = g0; g < g1; ++g) {
    const int64_t old = count[g], add = bcount[g], nw = old + add;
    tp += ceil_div(nw, kPageRows);
    np += ceil_div(nw, kPageRows) - ceil_div(old, kPageRows);
    ns += ceil_div(add, seg_rows);
    nt += add > 0;
  }
  int64_t o_tp = block_scan_incl(tp, sh) - tp;
  int64_t o_np = block_scan_incl(np, sh) - np;
  int64_t o_ns = block_scan_incl(ns, sh) - ns;
  int64_t o_nt = block_scan_incl(nt, sh) - nt;
  const int64_t pages_used = dev_ctr[1];
  for (int g = g0; g < g1; ++g) {
    const int64_t old = count[g], add = bcount[g], nw = old + add;
    page_off_new[g] = (int32_t)o_tp;
    first_new[g] = (int32_t)(pages_used + o_np);
    base[g] = (int32_t)old;
    o_tp += ceil_div(nw, kPageRows);
    o_np += ceil_div(nw, kPageRows) - ceil_div(old, kPageRows);
    if (add > 0) {
      const int32_t s0 = (int32_t)o_ns;
      for (int64_t r = old; r < nw; r += seg_rows) {
        segs[o_ns++] = KeySeg{g, (int32_t)r, (int32_t)min(nw, r + seg_rows), 0};
      }
      kgroups[o_nt++] = KeyGroup{g, s0, (int32_t)o_ns, (int32_t)nw, nw > 0 ? 1.0 / (double)nw : 0.0};
      count[g] = (int32_t)nw;
    }
    bcount[g] = 0;  // read for the last time: cleared for the next batch
  }
  if (threadIdx.x == 0) bcount[G + 1] = 0;
  // The last thread's running offsets are the totals.
  if (threadIdx.x == kLayoutThreads - 1) {
    page_off_new[G] = (int32_t)o_tp;
    meta[0] = (int32_t)o_ns;
    meta[1] = (int32_t)o_nt;
    *id_base = dev_ctr[0];
    dev_ctr[0] += rows;
    dev_ctr[1] = pages_used + o_np;
  }
  if (!fuse_scan && !fuse_copy) return;
  __syncthreads();  // base, page_off_new and first_new of every group are written
  for (int g = warp; g < G; g += kLayoutThreads / 32) {
    if (fuse_scan) chunk_scan_group(g, lane, hist, n_chunks, base);
    if (fuse_copy) page_copy_group(g, lane, page_off_cur, page_list_cur, page_off_new, first_new, page_list_new);
  }
}

// One warp: group g's page list in the new layout (its current pages, then
// its fresh ones).
__device__ void page_copy_group(int g, int lane, const int32_t *page_off_cur, const int32_t *page_list_cur,
                                const int32_t *page_off_new, const int32_t *first_new, int32_t *page_list_new) {
  const int32_t c0 = page_off_cur[g], n_old = page_off_cur[g + 1] - c0;
  const int32_t n0 = page_off_new[g], n_tot = page_off_new[g + 1] - n0;
  for (int32_t i = lane; i < n_tot; i += 32) {
    page_list_new[n0 + i] = i < n_old ? page_list_cur[c0 + i] : first_new[g] + (i - n_old);
  }
}

// One warp: hist[g][c] <- base[g] + sum_{c' < c} hist[g][c'].
__device__ void chunk_scan_group(int g, int lane, int32_t *hist, int64_t n_chunks, const int32_t *base) {
  int32_t *row = hist + (int64_t)g * n_chunks;
  int32_t running = base[g];
  for (int64_t c0 = 0; c0 < n_chunks; c0 += 32) {
    int64_t c = c0 + lane;
    int32_t v = c < n_chunks ? row[c] : 0;
    int32_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int32_t t = __shfl_up_sync(kFullMask, incl, o);
      if (lane >= o) incl += t;
    }
    if (c < n_chunks) row[c] = running + incl - v;
    running += __shfl_sync(kFullMask, incl, 31);
  }
}

// Per group (one warp each), for large layouts: the page list copy and, for a
// batch that passed the check, the chunk scan, in one launch.
__global__ void group_lists_kernel(int32_t G, const int32_t *__restrict__ page_off_cur,
                                   const int32_t *__restrict__ page_list_cur, const int32_t *__restrict__ page_off_new,
                                   const int32_t *__restrict__ first_new, int32_t *__restrict__ page_list_new,
                                   int do_copy, int32_t *__restrict__ hist, int64_t n_chunks, int do_scan,
                                   const int32_t *__restrict__ base, const int32_t *__restrict__ bad) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int g = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (g >= G) return;
  if (do_copy) page_copy_group(g, lane, page_off_cur, page_list_cur, page_off_new, first_new, page_list_new);
  if (do_scan && !*bad) chunk_scan_group(g, lane, hist, n_chunks, base);
}

// One warp per chunk walks its rows in order; rows of the same group take
// consecutive slots (stable), so pos[e] = slot of row e within its group.
__global__ void chunk_place_kernel(const int32_t *__restrict__ gid, const int32_t *__restrict__ ids, int64_t n,
                                   int64_t chunk, int64_t n_chunks, int32_t *__restrict__ hist,
                                   int32_t *__restrict__ pos, const int32_t *__restrict__ bad) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  if (*bad) return;
  int64_t c = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (c >= n_chunks) return;
  int64_t lo = c * chunk, hi = min(n, lo + chunk);
  unsigned lt = (1u << lane) - 1u;
  for (int64_t b0 = lo; b0 < hi; b0 += 32) {
    int64_t e = b0 + lane;
    unsigned act = __ballot_sync(kFullMask, e < hi);
    if (e < hi) {
      int32_t g = row_group(gid, ids, e);
      unsigned peers = __match_any_sync(act, g);
      int leader = __ffs(peers) - 1;
      int rank = __popc(peers & lt);
      int32_t old = 0;
      int32_t *slot = &hist[(int64_t)g * n_chunks + c];
      if (lane == leader) {
        old = *slot;
        *slot = old + __popc(peers);
      }
      old = __shfl_sync(act, old, leader);
      pos[e] = old + rank;
    }
    __syncwarp();
  }
}

// Chunks of 32 rows (appends): one block per chunk.  Its first warp takes
// the chunk's rows in order and gives each its slot as chunk_place_kernel
// does; then the block's eight warps copy the rows into their slots as
// place_rows_kernel does, four rows each.  (Every group id of the chunk is
// read before the barrier, so `assigned` may alias `gid`.)
constexpr int kPlaceWarps = 8;
__global__ void __launch_bounds__(kPlaceWarps * 32)
    place_chunk_kernel(const uint4 *__restrict__ src, const int32_t *gid, const int32_t *__restrict__ ids, int64_t n,
                       int64_t n_chunks, int32_t *__restrict__ hist, int vec_per_row,
                       const int32_t *__restrict__ page_list, const int32_t *__restrict__ page_off,
                       uint4 *__restrict__ pool, int32_t *__restrict__ slot_id, const int64_t *__restrict__ id_base,
                       int32_t *assigned, const int32_t *__restrict__ bad) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  __shared__ int32_t s_grp[32], s_pos[32];
  if (*bad) return;  // uniform over the grid
  const int64_t c = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t lo = c * 32, hi = min(n, lo + 32);
  if (warp == 0) {
    const int64_t e = lo + lane;
    const unsigned act = __ballot_sync(kFullMask, e < hi);
    if (e < hi) {
      const int32_t g = row_group(gid, ids, e);
      const unsigned peers = __match_any_sync(act, g);
      const int leader = __ffs(peers) - 1;
      const int rank = __popc(peers & ((1u << lane) - 1u));
      int32_t old = 0;
      int32_t *slot = &hist[(int64_t)g * n_chunks + c];
      if (lane == leader) {
        old = *slot;
        *slot = old + __popc(peers);
      }
      old = __shfl_sync(act, old, leader);
      s_grp[lane] = g;
      s_pos[lane] = old + rank;
    }
  }
  __syncthreads();
  const int rows = (int)(hi - lo);
  for (int i = warp; i < rows; i += kPlaceWarps) {
    const int64_t e = lo + i;
    const int32_t g = s_grp[i], p = s_pos[i];
    const int64_t page = page_list[page_off[g] + p / kPageRows];
    const int64_t sl = page * kPageRows + (p % kPageRows);
    const uint4 *s = src + e * vec_per_row;
    uint4 *dst = pool + sl * vec_per_row;
    for (int v = lane; v < vec_per_row; v += 32) dst[v] = s[v];
    if (lane == 0) {
      slot_id[sl] = (int32_t)(*id_base + e);
      if (assigned) assigned[e] = g;
    }
  }
}

// One warp per row: copy into its page slot, record its entry id (and, when
// asked, the group it joined).
__global__ void place_rows_kernel(const uint4 *__restrict__ src, const int32_t *gid, const int32_t *__restrict__ ids,
                                  const int32_t *__restrict__ pos, int64_t n, int vec_per_row,
                                  const int32_t *__restrict__ page_list, const int32_t *__restrict__ page_off,
                                  uint4 *__restrict__ pool, int32_t *__restrict__ slot_id,
                                  const int64_t *__restrict__ id_base, int32_t *assigned,
                                  const int32_t *__restrict__ bad) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  if (*bad) return;
  int64_t e = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (e >= n) return;  // uniform per warp
  // Lane 0 reads the group and hands it to the warp, so no lane reads gid[e]
  // after lane 0 may have overwritten it through `assigned`.
  int32_t g = lane == 0 ? row_group(gid, ids, e) : 0;
  g = __shfl_sync(kFullMask, g, 0);
  int32_t p = pos[e];
  int64_t page = page_list[page_off[g] + p / kPageRows];
  int64_t slot = page * kPageRows + (p % kPageRows);
  const uint4 *s = src + e * vec_per_row;
  uint4 *dst = pool + slot * vec_per_row;
  for (int v = lane; v < vec_per_row; v += 32) dst[v] = s[v];
  if (lane == 0) {
    slot_id[slot] = (int32_t)(*id_base + e);
    if (assigned) assigned[e] = g;  // after this row's own read of gid[e] (assigned may be gid)
  }
}


// partial[s][j] = sum over rows r0..r1-1 of group g of row[j], accumulated
// in fp32 with Kahan compensation and returned as fp64 (sum + compensation),
// so the key error does not grow with the segment length.  Rows are loaded
// eight at a time before any is added, so the loads of a thread overlap.
template <typename T>
__global__ void key_partial_kernel(const T *__restrict__ pool, int32_t d,
                                   const int32_t *__restrict__ page_list,
                                   const int32_t *__restrict__ page_off,
                                   const KeySeg *__restrict__ segs, const int32_t *__restrict__ n_segs,
                                   double *__restrict__ partial) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  constexpr int kBatch = 8;
  if ((int)blockIdx.x >= *n_segs) return;  // the grid covers the host's bound on the segments
  const KeySeg sg = segs[blockIdx.x];
  const int j0 = (blockIdx.y * blockDim.x + threadIdx.x) * 8;
  if (j0 >= d) return;
  float acc[8], comp[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = comp[i] = 0.f;
  const int32_t *pages = page_list + page_off[sg.g];
  for (int r = sg.r0; r < sg.r1; r += kBatch) {
    float x[kBatch][8];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int rr = min(r + u, sg.r1 - 1);  // rows past the segment are loaded but not added
      const int64_t slot = (int64_t)pages[rr / kPageRows] * kPageRows + (rr % kPageRows);
      const T *row = pool + slot * d + j0;
      if constexpr (sizeof(T) == 2) {
        const uint4 v = *reinterpret_cast<const uint4 *>(row);
        x[u][0] = bf16lo(v.x); x[u][1] = bf16hi(v.x); x[u][2] = bf16lo(v.y); x[u][3] = bf16hi(v.y);
        x[u][4] = bf16lo(v.z); x[u][5] = bf16hi(v.z); x[u][6] = bf16lo(v.w); x[u][7] = bf16hi(v.w);
      } else {
        const float4 a = *reinterpret_cast<const float4 *>(row);
        const float4 b = *reinterpret_cast<const float4 *>(row + 4);
        x[u][0] = a.x; x[u][1] = a.y; x[u][2] = a.z; x[u][3] = a.w;
        x[u][4] = b.x; x[u][5] = b.y; x[u][6] = b.z; x[u][7] = b.w;
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      if (r + u < sg.r1) {  // uniform across the block
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float y = x[u][i] - comp[i];
          const float t = acc[i] + y;
          comp[i] = (t - acc[i]) - y;
          acc[i] = t;
        }
      }
    }
  }
  double *out = partial + (int64_t)blockIdx.x * d + j0;
#pragma unroll
  for (int i = 0; i < 8; ++i) out[i] = (double)acc[i] - (double)comp[i];
}

// csum[g] += partials in segment order; refresh the fp32 mean and its bf16
// hi/lo split for the group.
// Also writes the host mirror slot (pinned host memory, mapped): the entry
// count and every group's size after the batch, one group per block of the
// first column range, so that no copy follows the append in the stream.
__global__ void key_finalize_kernel(const KeyGroup *__restrict__ groups, const int32_t *__restrict__ n_groups,
                                    const double *__restrict__ partial, int32_t d,
                                    double *__restrict__ csum, float *__restrict__ cent,
                                    __nv_bfloat16 *__restrict__ hi, __nv_bfloat16 *__restrict__ lo,
                                    const int32_t *__restrict__ count, const int64_t *__restrict__ dev_ctr,
                                    char *mirror, int32_t *__restrict__ bad, int32_t *__restrict__ hist,
                                    int64_t hist_len) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  // The batch's remaining counters (read by nothing after the row placement):
  // the check flag and the (group, chunk) counts, cleared for the next batch.
  {
    const int64_t t0 = ((int64_t)blockIdx.y * gridDim.x + blockIdx.x) * blockDim.x + threadIdx.x;
    const int64_t nt = (int64_t)gridDim.x * gridDim.y * blockDim.x;
    for (int64_t t = t0; t < hist_len; t += nt) hist[t] = 0;
    if (t0 == 0) *bad = 0;
  }
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    if (blockIdx.x == 0) *reinterpret_cast<volatile int64_t *>(mirror) = dev_ctr[0];
    reinterpret_cast<volatile int32_t *>(mirror + sizeof(int64_t))[blockIdx.x] = count[blockIdx.x];
    __threadfence_system();
  }
  if ((int)blockIdx.x >= *n_groups) return;  // the grid covers every group
  KeyGroup kg = groups[blockIdx.x];
  // The group's fp64 reciprocal comes from the layout block (fp64
  // arithmetic is slow on this part, a division most of all); the mean is
  // then rounded to fp32 and split in fp32: hi = bf16(mean), lo = bf16(mean - hi).
  const double inv = kg.inv;
  for (int j = blockIdx.y * blockDim.x + threadIdx.x; j < d; j += gridDim.y * blockDim.x) {
    // The segments' partial sums added in segment order, loaded eight at a
    // time so that a group of many segments is not one load per step.
    double add = 0.0;
    for (int s0 = kg.seg0; s0 < kg.seg1; s0 += 8) {
      double v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = s0 + u < kg.seg1 ? partial[(int64_t)(s0 + u) * d + j] : 0.0;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (s0 + u < kg.seg1) add += v[u];
      }
    }
    int64_t o = (int64_t)kg.g * d + j;
    double sum = csum[o] + add;
    csum[o] = sum;
    const float mean = (float)(sum * inv);
    cent[o] = mean;
    const __nv_bfloat16 h = __float2bfloat16_rn(mean);
    hi[o] = h;
    lo[o] = __float2bfloat16_rn(mean - __bfloat162float(h));
  }
}

}  // namespace

htam_status ensure_scratch(htam_memory *m, size_t bytes) {
  if (bytes <= m->scratch_bytes) return HTAM_OK;
  if (m->scratch) {
    cudaFree(m->scratch);  // implicit device synchronisation: no queued work still uses it
    m->scratch = nullptr;
    m->scratch_bytes = 0;
  }
  // Half again as much as asked: a memory that grows by appends asks for a
  // little more scratch every query, and each reallocation costs a device
  // synchronisation (cudaFree) and an allocation.
  size_t want = std::max(bytes + bytes / 2, size_t(1) << 20);
  if (cudaMalloc(&m->scratch, want) != cudaSuccess) {
    cudaGetLastError();
    m->scratch = nullptr;
    return HTAM_ENOMEM;
  }
  m->scratch_bytes = want;
  return HTAM_OK;
}

htam_status refresh_mirror(htam_memory *m, bool wait) {
  if (m->mirror_seq == m->append_seq) return HTAM_OK;
  constexpr int S = htam_memory::kMirrorSlots;
  if (wait) {
    const int newest = (int)(m->append_seq % S);
    HTAM_CK(cudaEventSynchronize(m->mirror_ev[newest]));
  }
  // The newest slot whose copies have landed.
  for (int64_t q = m->append_seq; q > m->mirror_seq && q > m->append_seq - S; --q) {
    const int slot = (int)(q % S);
    if (m->slot_seq[slot] != q) continue;
    cudaError_t e = cudaEventQuery(m->mirror_ev[slot]);
    if (e == cudaErrorNotReady) continue;
    if (e != cudaSuccess) {
      set_last_error("cudaEventQuery", e);
      return HTAM_ECUDA;
    }
    const char *p = static_cast<const char *>(m->h_pin) + slot * m->pin_slot_bytes;
    const int64_t n_dev = *reinterpret_cast<const int64_t *>(p);
    const int32_t *c = reinterpret_cast<const int32_t *>(p + sizeof(int64_t));
    for (int32_t g = 0; g < m->n_groups; ++g) m->h_count[g] = c[g];
    m->mirror_seq = q;
    m->rows_pending = m->rows_issued - m->slot_rows_issued[slot];
    m->n = n_dev + m->rows_pending;
    return HTAM_OK;
  }
  return HTAM_OK;
}

// Files `count` rows under their groups and updates the keys of the groups
// they join (the memory update of Eq. 15), entirely on the device: the batch's
// group sizes, the nearest-key choice for rows given -1 (appends only), the
// page layout, the stable slot order and the key sums are all computed by
// kernels queued on `st`, with no host round trip.  Group ids are checked on
// the device: a bad batch (an id out of range, or -1 with no non-empty group
// to join) is skipped by every kernel after the check and recorded in status
// bit 1, leaving the memory unchanged.  `build` (the first batch of a new
// memory) takes no -1 ids.
static htam_status add_rows(htam_memory *m, const void *entries, const int32_t *gid, int64_t count,
                            int32_t *assigned, cudaStream_t st, bool build) {
  if (count == 0) return HTAM_OK;
  PdlScope pdl(m->pdl != 0);
  const int32_t G = m->n_groups, d = m->d;

  // Chunking of the stable sort: at most ~16M (group, chunk) counters; one
  // warp-wide step per chunk for batches of up to 64K rows (an append), so
  // the placing warps do not walk long chunks one after another.
  int64_t chunk = std::max<int64_t>(count <= 65536 ? 32 : 256, ceil_div((int64_t)count * G, int64_t(1) << 24));
  chunk = ceil_div(chunk, 32) * 32;
  int64_t n_chunks = ceil_div(count, chunk);

  // Key segments: at most count/seg_rows + (touched groups) of them.
  const int seg_rows = key_seg_rows(count);
  int64_t max_segs = std::min<int64_t>(count, count / seg_rows + G + 1);

  size_t need = Carver::round(sizeof(int32_t) * 4) + Carver::round(sizeof(int64_t)) +
                (build ? 0 : Carver::round(sizeof(int32_t) * count)) + Carver::round(sizeof(int32_t) * count) +
                Carver::round(sizeof(KeySeg) * max_segs) + Carver::round(sizeof(KeyGroup) * G) +
                2 * Carver::round(sizeof(int32_t) * G) + Carver::round(sizeof(double) * (size_t)max_segs * d) + 4096;
  htam_status s = ensure_scratch(m, need);
  if (s != HTAM_OK) return s;
  // The batch counters live in a buffer of the memory object that is zero
  // between batches: the batch's group counts, the check flag, the count of
  // rows without a group, then the (group, chunk) counts of the stable sort.
  // The layout block clears the first and the last of the three, the key
  // finalisation the flag and the (group, chunk) counts, so no memset
  // starts a batch; a batch that stopped early leaves them marked dirty and
  // the next one clears them first.
  const int64_t hist_off = ceil_div(G + 2, 64) * 64;
  const int64_t n_ctr = hist_off + (int64_t)G * n_chunks;
  if (n_ctr > m->batch_ctr_len) {
    if (m->batch_ctr) cudaFree(m->batch_ctr);  // synchronises: no queued work still uses it
    m->batch_ctr = nullptr;
    m->batch_ctr_len = 0;
    const int64_t want = n_ctr + n_ctr / 2;
    if (cudaMalloc(&m->batch_ctr, sizeof(int32_t) * want) != cudaSuccess) {
      cudaGetLastError();
      m->batch_ctr = nullptr;
      return HTAM_ENOMEM;
    }
    m->batch_ctr_len = want;
    m->batch_dirty = true;
  }
  Carver cv(m->scratch);
  int32_t *bcount = m->batch_ctr;              // [G] counts, bad flag, rows without a group
  int32_t *meta = cv.take<int32_t>(4);         // key segments, touched groups
  int64_t *id_base = cv.take<int64_t>(1);
  int32_t *ids = build ? nullptr : cv.take<int32_t>(count);  // groups chosen for rows given -1
  int32_t *pos = cv.take<int32_t>(count);
  int32_t *hist = bcount + hist_off;
  KeySeg *segs = cv.take<KeySeg>(max_segs);
  KeyGroup *kgroups = cv.take<KeyGroup>(G);
  int32_t *first_new = cv.take<int32_t>(G);
  int32_t *base = cv.take<int32_t>(G);
  double *partial = cv.take<double>((size_t)max_segs * d);
  int32_t *bad = bcount + G;

  PhaseMark mark(m, st);
  mark.begin(HTAM_PHASE_APPEND);

  // 1. Per-group and per-(group, chunk) counts of the batch and the
  //    group-id range check.
  if (m->batch_dirty) HTAM_CK(cudaMemsetAsync(bcount, 0, sizeof(int32_t) * m->batch_ctr_len, st));
  m->batch_dirty = true;  // until the key finalisation below is queued
  {
    const int blocks = (int)std::min<int64_t>(ceil_div(count, 256), 4096);
    launch_kernel(count_groups_kernel, blocks, 256, 0, st, gid, count, G, build ? 0 : 1, bcount, bad, bcount + G + 1,
                  hist, chunk, n_chunks);
    HTAM_CK_LAUNCH("count_groups_kernel");
    mark.launched();
  }
  // 2. Rows without a group join the group whose key scores highest against
  //    them, by the keys as they stand before this call.  The kernels run
  //    only when the count above found such rows.
  if (!build) {
    s = assign_unassigned(m, entries, gid, count, bcount + G + 1, ids, bcount, bad, hist, chunk, n_chunks, st,
                          &mark);
    if (s != HTAM_OK) return s;
  }
  // 3. Page layout, key segments and new sizes; then the page lists and the
  //    scan of the (group, chunk) counts from each group's old size (in the
  //    same block when they are small, one warp per group, else by kernels
  //    of their own).
  // (One block walks each warp's groups one after another, so this pays
  // only for a few counters and pages; the 512-group streaming workload
  // runs faster with the separate kernels.)
  const bool fuse_scan = (int64_t)G * n_chunks <= 2048;
  const bool fuse_copy = m->n_pages_max <= 2048;
  launch_kernel(layout_kernel, 1, kLayoutThreads, 0, st, G, count, seg_rows, bcount, bad, m->count, m->page_off,
                m->page_off_alt, first_new, base, segs, kgroups, meta, id_base, m->dev_ctr, m->status,
                fuse_scan ? 1 : 0, hist, n_chunks, fuse_copy ? 1 : 0, m->page_list, m->page_list_alt);
  HTAM_CK_LAUNCH("layout_kernel");
  mark.launched();
  // 4. The page lists of the new layout and the scan of the (group, chunk)
  //    counts from each group's old size, one warp per group, when the
  //    layout block did not do them.
  if (!fuse_copy || !fuse_scan) {
    launch_kernel(group_lists_kernel, (unsigned)ceil_div((int64_t)G * 32, 256), 256, 0, st, G, m->page_off,
                  m->page_list, m->page_off_alt, first_new, m->page_list_alt, fuse_copy ? 0 : 1, hist, n_chunks,
                  fuse_scan ? 0 : 1, base, bad);
    HTAM_CK_LAUNCH("group_lists_kernel");
    mark.launched();
  }

  // 5. Stable slot assignment (pos[e] = old size of its group + rank among
  //    earlier rows of the batch with the same group), then the rows copied
  //    into their slots: one launch for chunks of 32 rows (appends), two
  //    for the long chunks of large builds.
  int vec_per_row = d * m->elem_bytes / 16;
  if (chunk == 32) {
    launch_kernel(place_chunk_kernel, (unsigned)n_chunks, kPlaceWarps * 32, 0, st,
                  static_cast<const uint4 *>(entries), gid, ids, count, n_chunks, hist, vec_per_row,
                  m->page_list_alt, m->page_off_alt, static_cast<uint4 *>(m->pool), m->slot_id, id_base, assigned,
                  bad);
    HTAM_CK_LAUNCH("place_chunk_kernel");
    mark.launched();
  } else {
    launch_kernel(chunk_place_kernel, (unsigned)ceil_div(n_chunks * 32, 256), 256, 0, st, gid, ids, count, chunk,
                  n_chunks, hist, pos, bad);
    HTAM_CK_LAUNCH("chunk_place_kernel");
    launch_kernel(place_rows_kernel, (unsigned)ceil_div(count * 32, 256), 256, 0, st,
                  static_cast<const uint4 *>(entries), gid, ids, pos, count, vec_per_row, m->page_list_alt,
                  m->page_off_alt, static_cast<uint4 *>(m->pool), m->slot_id, id_base, assigned, bad);
    HTAM_CK_LAUNCH("place_rows_kernel");
    mark.launched(2);
  }

  // 6. Keys of the touched groups.
  {
    // 8 columns per thread: 128 threads cover d = 1,024.
    const int kp_threads = (int)std::min<int64_t>(256, ceil_div(ceil_div(d, 8), 32) * 32);
    dim3 grid((unsigned)max_segs, (unsigned)ceil_div(d, kp_threads * 8));
    if (m->dtype == HTAM_BF16) {
      launch_kernel(key_partial_kernel<__nv_bfloat16>, grid, kp_threads, 0, st, static_cast<const __nv_bfloat16 *>(m->pool), d,
                                                              m->page_list_alt, m->page_off_alt, segs, meta,
                                                              partial);
    } else {
      launch_kernel(key_partial_kernel<float>, grid, kp_threads, 0, st, static_cast<const float *>(m->pool), d, m->page_list_alt,
                                                      m->page_off_alt, segs, meta, partial);
    }
    HTAM_CK_LAUNCH("key_partial_kernel");
    dim3 g2((unsigned)G, (unsigned)std::min<int64_t>(ceil_div(d, 256), 16));
    const int slot = (int)((m->append_seq + 1) % htam_memory::kMirrorSlots);
    char *mirror = static_cast<char *>(m->d_pin) + slot * m->pin_slot_bytes;
    launch_kernel(key_finalize_kernel, g2, 256, 0, st, kgroups, meta + 1, partial, d, m->csum, m->cent, m->cent_hi,
                  m->cent_lo, m->count, m->dev_ctr, mirror, bad, hist, (int64_t)G * n_chunks);
    HTAM_CK_LAUNCH("key_finalize_kernel");
    m->batch_dirty = false;
    mark.launched(2);
  }

  // 7. The new layout is current from here on in stream order; the sizes
  //    and the entry count go to the next mirror slot.
  std::swap(m->page_list, m->page_list_alt);
  std::swap(m->page_off, m->page_off_alt);
  m->append_seq += 1;
  m->rows_issued += count;
  m->rows_pending += count;
  m->n += count;
  // (key_finalize_kernel wrote the slot; its event marks it complete.)
  const int slot = (int)(m->append_seq % htam_memory::kMirrorSlots);
  HTAM_CK(cudaEventRecord(m->mirror_ev[slot], st));
  m->slot_seq[slot] = m->append_seq;
  m->slot_rows_issued[slot] = m->rows_issued;
  m->last_stream = st;
  mark.end();
  return HTAM_OK;
}

void free_impl(htam_memory *m) {
  if (!m) return;
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(m->device);
  cudaFree(m->pool);
  cudaFree(m->slot_id);
  cudaFree(m->page_list);
  cudaFree(m->page_off);
  cudaFree(m->page_list_alt);
  cudaFree(m->page_off_alt);
  cudaFree(m->dev_ctr);
  cudaFree(m->batch_ctr);
  cudaFree(m->qbits);
  if (m->h_pin) cudaFreeHost(m->h_pin);
  for (cudaEvent_t e : m->mirror_ev) {
    if (e) cudaEventDestroy(e);
  }
  if (m->ev_fork) cudaEventDestroy(m->ev_fork);
  if (m->ev_join) cudaEventDestroy(m->ev_join);
  if (m->side) cudaStreamDestroy(m->side);
  cudaFree(m->count);
  cudaFree(m->csum);
  cudaFree(m->cent);
  cudaFree(m->cent_hi);
  cudaFree(m->cent_lo);
  cudaFree(m->status);
  cudaFree(m->scratch);
  cudaFree(m->stage);
  cudaFree(m->prefix_buf);
  cudaFree(m->assign_buf);
  for (cudaEvent_t e : m->ev_pool) cudaEventDestroy(e);
  cudaGetLastError();
  cudaSetDevice(prev);
  delete m;
}

htam_status build_impl(const void *entries, const int32_t *gid, int64_t n, int32_t d,
                       int32_t n_groups, htam_dtype dtype, int64_t capacity, cudaStream_t st,
                       htam_memory **out) {
  htam_memory *m = new (std::nothrow) htam_memory();
  if (!m) return HTAM_ENOMEM;
  HTAM_CK(cudaGetDevice(&m->device));
  HTAM_CK(cudaDeviceGetAttribute(&m->sm_count, cudaDevAttrMultiProcessorCount, m->device));
  m->d = d;
  // Buckets of two or more queries go to the tensor cores: a padded 128-row
  // tile still streams its entries at HBM speed, while the CUDA cores are
  // compute-bound with several queries per row for d <= 2048 and, for
  // longer rows, score at most two queries per pass (the rest re-read the
  // rows).  Measured: 2 is the fastest threshold on every workload tried.
  m->tc_min = 2;
  m->n_groups = n_groups;
  m->dtype = dtype;
  m->elem_bytes = dtype == HTAM_BF16 ? 2 : 4;
  m->capacity = capacity;
  m->n_pages_max = ceil_div(capacity, kPageRows) + n_groups;
  m->h_count.assign(n_groups, 0);

  auto fail = [&](htam_status s) {
    free_impl(m);
    return s;
  };
  size_t pool_bytes = (size_t)m->n_pages_max * kPageRows * d * m->elem_bytes;
  size_t gd = (size_t)n_groups * d;
  if (cudaMalloc(&m->pool, pool_bytes) != cudaSuccess ||
      cudaMalloc(&m->slot_id, sizeof(int32_t) * m->n_pages_max * kPageRows) != cudaSuccess ||
      cudaMalloc(&m->page_list, sizeof(int32_t) * m->n_pages_max) != cudaSuccess ||
      cudaMalloc(&m->page_off, sizeof(int32_t) * (n_groups + 1)) != cudaSuccess ||
      cudaMalloc(&m->page_list_alt, sizeof(int32_t) * m->n_pages_max) != cudaSuccess ||
      cudaMalloc(&m->page_off_alt, sizeof(int32_t) * (n_groups + 1)) != cudaSuccess ||
      cudaMalloc(&m->dev_ctr, sizeof(int64_t) * 2) != cudaSuccess ||
      cudaMalloc(&m->count, sizeof(int32_t) * n_groups) != cudaSuccess ||
      cudaMalloc(&m->csum, sizeof(double) * gd) != cudaSuccess ||
      cudaMalloc(&m->cent, sizeof(float) * gd) != cudaSuccess ||
      cudaMalloc(&m->cent_hi, sizeof(__nv_bfloat16) * gd) != cudaSuccess ||
      cudaMalloc(&m->cent_lo, sizeof(__nv_bfloat16) * gd) != cudaSuccess ||
      cudaMalloc(&m->status, sizeof(unsigned int)) != cudaSuccess) {
    cudaGetLastError();
    return fail(HTAM_ENOMEM);
  }
  // Pinned mirror slots (entry count + group sizes) and their events.
  m->pin_slot_bytes = Carver::round(sizeof(int64_t) + sizeof(int32_t) * (size_t)n_groups);
  if (cudaMallocHost(&m->h_pin, m->pin_slot_bytes * htam_memory::kMirrorSlots) != cudaSuccess) {
    cudaGetLastError();
    m->h_pin = nullptr;
    return fail(HTAM_ENOMEM);
  }
  if (cudaHostGetDevicePointer(&m->d_pin, m->h_pin, 0) != cudaSuccess) {
    set_last_error("cudaHostGetDevicePointer", cudaGetLastError());
    return fail(HTAM_ECUDA);
  }
  for (cudaEvent_t &e : m->mirror_ev) {
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      e = nullptr;
      return fail(HTAM_ECUDA);
    }
  }
  // Empty rows are zero (never NaN), empty slots have id -1, keys start at 0.
  if (cudaMemsetAsync(m->pool, 0, pool_bytes, st) != cudaSuccess ||
      cudaMemsetAsync(m->slot_id, 0xff, sizeof(int32_t) * m->n_pages_max * kPageRows, st) != cudaSuccess ||
      cudaMemsetAsync(m->page_off, 0, sizeof(int32_t) * (n_groups + 1), st) != cudaSuccess ||
      cudaMemsetAsync(m->page_off_alt, 0, sizeof(int32_t) * (n_groups + 1), st) != cudaSuccess ||
      cudaMemsetAsync(m->dev_ctr, 0, sizeof(int64_t) * 2, st) != cudaSuccess ||
      cudaMemsetAsync(m->count, 0, sizeof(int32_t) * n_groups, st) != cudaSuccess ||
      cudaMemsetAsync(m->csum, 0, sizeof(double) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->cent, 0, sizeof(float) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->cent_hi, 0, sizeof(__nv_bfloat16) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->cent_lo, 0, sizeof(__nv_bfloat16) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->status, 0, sizeof(unsigned int), st) != cudaSuccess) {
    set_last_error("cudaMemsetAsync", cudaGetLastError());
    return fail(HTAM_ECUDA);
  }
  // The build is the one synchronous batch: a group id out of range fails
  // the call (and frees the memory) instead of being reported later.
  // The check's outcome is status bit 1 (set by the layout block for a
  // rejected batch).
  htam_status s = add_rows(m, entries, gid, n, nullptr, st, /*build=*/true);
  if (s != HTAM_OK) return fail(s);
  unsigned h_status = 0;
  if (cudaMemcpyAsync(&h_status, m->status, sizeof h_status, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess) {
    set_last_error("htam_build_memory: reading the group-id check", cudaGetLastError());
    return fail(HTAM_ECUDA);
  }
  if (h_status & 2u) return fail(HTAM_EINVAL);
  s = refresh_mirror(m, true);
  if (s != HTAM_OK) return fail(s);
  *out = m;
  return HTAM_OK;
}

htam_status append_impl(htam_memory *m, const void *entries, const int32_t *gid, int64_t count,
                        int32_t *assigned, cudaStream_t st) {
  if (m->n + count > m->capacity) {
    // The host's count may still include appends the device rejected: look
    // at the device's before refusing.
    htam_status s = refresh_mirror(m, true);
    if (s != HTAM_OK) return s;
    if (m->n + count > m->capacity) return HTAM_ECAPACITY;
  }
  return add_rows(m, entries, gid, count, assigned, st, /*build=*/false);
}

}  // namespace htam
