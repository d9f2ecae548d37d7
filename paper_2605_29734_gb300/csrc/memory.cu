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

constexpr int kKeySegRowsMin = 64;     // rows per key partial-sum segment: at least this,
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

// Per-group counts of a batch; ids of -1 (no group given) are counted apart,
// any other id outside [0, n_groups) sets `bad`.
__global__ void count_groups_kernel(const int32_t *__restrict__ gid, int64_t n, int32_t n_groups,
                                    int32_t *__restrict__ counts, int32_t *__restrict__ bad,
                                    int32_t *__restrict__ unassigned) {
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n;
       e += (int64_t)gridDim.x * blockDim.x) {
    int32_t g = gid[e];
    if (g == -1) {
      atomicAdd(unassigned, 1);
    } else if (g < 0 || g >= n_groups) {
      atomicOr(bad, 1);
    } else {
      atomicAdd(&counts[g], 1);
    }
  }
}

// hist[g * n_chunks + c] = number of rows of group g in chunk c.
__global__ void chunk_hist_kernel(const int32_t *__restrict__ gid, int64_t n, int64_t chunk,
                                  int64_t n_chunks, int32_t *__restrict__ hist) {
  int64_t c = blockIdx.x;
  int64_t lo = c * chunk, hi = min(n, lo + chunk);
  for (int64_t e = lo + threadIdx.x; e < hi; e += blockDim.x) {
    atomicAdd(&hist[(int64_t)gid[e] * n_chunks + c], 1);
  }
}

// Per group (one warp each): hist[g][c] <- base[g] + sum_{c' < c} hist[g][c'].
__global__ void chunk_scan_kernel(int32_t *__restrict__ hist, int64_t n_chunks, int32_t n_groups,
                                  const int32_t *__restrict__ base) {
  int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (warp >= n_groups) return;
  int32_t *row = hist + (int64_t)warp * n_chunks;
  int32_t running = base[warp];
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

// One warp per chunk walks its rows in order; rows of the same group take
// consecutive slots (stable), so pos[e] = slot of row e within its group.
__global__ void chunk_place_kernel(const int32_t *__restrict__ gid, int64_t n, int64_t chunk,
                                   int64_t n_chunks, int32_t *__restrict__ hist,
                                   int32_t *__restrict__ pos) {
  int64_t c = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (c >= n_chunks) return;
  int64_t lo = c * chunk, hi = min(n, lo + chunk);
  unsigned lt = (1u << lane) - 1u;
  for (int64_t b0 = lo; b0 < hi; b0 += 32) {
    int64_t e = b0 + lane;
    unsigned act = __ballot_sync(kFullMask, e < hi);
    if (e < hi) {
      int32_t g = gid[e];
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

// One warp per row: copy into its page slot, record its entry id.
__global__ void place_rows_kernel(const uint4 *__restrict__ src, const int32_t *__restrict__ gid,
                                  const int32_t *__restrict__ pos, int64_t n, int vec_per_row,
                                  const int32_t *__restrict__ page_list,
                                  const int32_t *__restrict__ page_off, uint4 *__restrict__ pool,
                                  int32_t *__restrict__ slot_id, int64_t id_base) {
  int64_t e = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  int lane = threadIdx.x & 31;
  if (e >= n) return;
  int32_t g = gid[e];
  int32_t p = pos[e];
  int64_t page = page_list[page_off[g] + p / kPageRows];
  int64_t slot = page * kPageRows + (p % kPageRows);
  const uint4 *s = src + e * vec_per_row;
  uint4 *dst = pool + slot * vec_per_row;
  for (int v = lane; v < vec_per_row; v += 32) dst[v] = s[v];
  if (lane == 0) slot_id[slot] = (int32_t)(id_base + e);
}

struct KeySeg {
  int32_t g, r0, r1, pad;
};
struct KeyGroup {
  int32_t g, seg0, seg1, count;
};

// partial[s][j] = sum over rows r0..r1-1 of group g of row[j], accumulated
// in fp32 with Kahan compensation and returned as fp64 (sum + compensation),
// so the key error does not grow with the segment length.  Rows are loaded
// eight at a time before any is added, so the loads of a thread overlap.
template <typename T>
__global__ void key_partial_kernel(const T *__restrict__ pool, int32_t d,
                                   const int32_t *__restrict__ page_list,
                                   const int32_t *__restrict__ page_off,
                                   const KeySeg *__restrict__ segs, double *__restrict__ partial) {
  constexpr int kBatch = 8;
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
__global__ void key_finalize_kernel(const KeyGroup *__restrict__ groups,
                                    const double *__restrict__ partial, int32_t d,
                                    double *__restrict__ csum, float *__restrict__ cent,
                                    __nv_bfloat16 *__restrict__ hi, __nv_bfloat16 *__restrict__ lo) {
  KeyGroup kg = groups[blockIdx.x];
  for (int j = blockIdx.y * blockDim.x + threadIdx.x; j < d; j += gridDim.y * blockDim.x) {
    double add = 0.0;
    for (int s = kg.seg0; s < kg.seg1; ++s) add += partial[(int64_t)s * d + j];
    int64_t o = (int64_t)kg.g * d + j;
    double sum = csum[o] + add;
    csum[o] = sum;
    double mean = kg.count > 0 ? sum / (double)kg.count : 0.0;
    cent[o] = (float)mean;
    __nv_bfloat16 h = __double2bfloat16(mean);
    hi[o] = h;
    lo[o] = __double2bfloat16(mean - (double)__bfloat162float(h));
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

// Files `count` rows (ids id_base..) under their groups and updates the keys
// of the groups they join.  Arguments are already validated except the group
// id range, which is checked on the device before anything is written.
static htam_status add_rows(htam_memory *m, const void *entries, const int32_t *gid, int64_t count,
                            int32_t *assigned, cudaStream_t st) {
  if (count == 0) return HTAM_OK;
  const int32_t G = m->n_groups, d = m->d;

  // Chunking of the stable sort: at most ~16M (group, chunk) counters.
  int64_t chunk = std::max<int64_t>(256, ceil_div((int64_t)count * G, int64_t(1) << 24));
  chunk = ceil_div(chunk, 32) * 32;
  int64_t n_chunks = ceil_div(count, chunk);

  // Key segments need the final layout; their number is bounded by
  // count/seg_rows + number of groups.
  const int seg_rows = key_seg_rows(count);
  int64_t max_segs = count / seg_rows + G + 1;

  size_t need = Carver::round(sizeof(int32_t) * (G + 2)) + Carver::round(sizeof(int32_t) * count) +
                Carver::round(sizeof(int32_t) * (size_t)G * n_chunks) +
                Carver::round(sizeof(KeySeg) * max_segs) + Carver::round(sizeof(KeyGroup) * G) +
                Carver::round(sizeof(double) * (size_t)max_segs * d) + 4096;
  htam_status s = ensure_scratch(m, need);
  if (s != HTAM_OK) return s;
  Carver cv(m->scratch);
  int32_t *bcount = cv.take<int32_t>(G + 2);  // [G] counts, bad flag, rows without a group
  int32_t *pos = cv.take<int32_t>(count);
  int32_t *hist = cv.take<int32_t>((size_t)G * n_chunks);
  KeySeg *segs = cv.take<KeySeg>(max_segs);
  KeyGroup *kgroups = cv.take<KeyGroup>(G);
  double *partial = cv.take<double>((size_t)max_segs * d);

  PhaseMark mark(m, st);
  mark.begin(HTAM_PHASE_APPEND);

  // 1. Per-group counts of the batch and the group-id range check.
  std::vector<int32_t> h_b(G + 2);
  auto count_batch = [&](const int32_t *ids) -> htam_status {
    HTAM_CK(cudaMemsetAsync(bcount, 0, sizeof(int32_t) * (G + 2), st));
    int blocks = (int)std::min<int64_t>(ceil_div(count, 256), 4096);
    count_groups_kernel<<<blocks, 256, 0, st>>>(ids, count, G, bcount, bcount + G, bcount + G + 1);
    HTAM_CK_LAUNCH("count_groups_kernel");
    mark.launched();
    HTAM_CK(cudaMemcpyAsync(h_b.data(), bcount, sizeof(int32_t) * (G + 2), cudaMemcpyDeviceToHost, st));
    HTAM_CK(cudaStreamSynchronize(st));
    return HTAM_OK;
  };
  s = count_batch(gid);
  if (s != HTAM_OK) return s;
  if (h_b[G] != 0) return HTAM_EINVAL;
  if (h_b[G + 1] > 0) {
    // Rows without a group join the group whose key scores highest against
    // them, by the keys as they stand before this call (none: EINVAL).
    bool any = false;
    for (int64_t c : m->h_count) any |= c > 0;
    if (!any) return HTAM_EINVAL;
    const int32_t *ids = nullptr;
    s = assign_nearest(m, entries, gid, count, assigned, &ids, st, &mark);
    if (s != HTAM_OK) return s;
    gid = ids;
    s = count_batch(gid);
    if (s != HTAM_OK) return s;
  } else if (assigned && assigned != gid) {
    HTAM_CK(cudaMemcpyAsync(assigned, gid, sizeof(int32_t) * count, cudaMemcpyDeviceToDevice, st));
  }

  // 2. Page layout on the host.
  std::vector<int64_t> new_count(G);
  int64_t new_pages = 0;
  for (int32_t g = 0; g < G; ++g) {
    new_count[g] = m->h_count[g] + h_b[g];
    new_pages += ceil_div(new_count[g], kPageRows) - ceil_div(m->h_count[g], kPageRows);
  }
  if (m->n + count > m->capacity || m->n_pages_used + new_pages > m->n_pages_max) {
    return HTAM_ECAPACITY;
  }
  // Every check has passed: from here on the layout is extended in place.
  std::vector<std::vector<int32_t>> &pages = m->h_pages;
  int64_t next_page = m->n_pages_used;
  std::vector<int32_t> h_off(G + 1), h_list;
  h_list.reserve((size_t)(m->n_pages_used + new_pages));
  for (int32_t g = 0; g < G; ++g) {
    int64_t want = ceil_div(new_count[g], kPageRows);
    while ((int64_t)pages[g].size() < want) pages[g].push_back((int32_t)next_page++);
    h_off[g] = (int32_t)h_list.size();
    h_list.insert(h_list.end(), pages[g].begin(), pages[g].end());
  }
  h_off[G] = (int32_t)h_list.size();

  // Key segments over the new rows of every touched group.
  std::vector<KeySeg> h_segs;
  std::vector<KeyGroup> h_kg;
  for (int32_t g = 0; g < G; ++g) {
    if (h_b[g] == 0) continue;
    KeyGroup kg{g, (int32_t)h_segs.size(), 0, (int32_t)new_count[g]};
    for (int64_t r = m->h_count[g]; r < new_count[g]; r += seg_rows) {
      h_segs.push_back(KeySeg{g, (int32_t)r, (int32_t)std::min<int64_t>(new_count[g], r + seg_rows), 0});
    }
    kg.seg1 = (int32_t)h_segs.size();
    h_kg.push_back(kg);
  }

  // From here on the memory is modified.  Upload the layout (stream
  // ordered after any earlier query on this stream).
  HTAM_CK(cudaMemcpyAsync(m->page_off, h_off.data(), sizeof(int32_t) * (G + 1), cudaMemcpyHostToDevice, st));
  if (!h_list.empty()) {
    HTAM_CK(cudaMemcpyAsync(m->page_list, h_list.data(), sizeof(int32_t) * h_list.size(),
                            cudaMemcpyHostToDevice, st));
  }
  HTAM_CK(cudaMemcpyAsync(segs, h_segs.data(), sizeof(KeySeg) * h_segs.size(), cudaMemcpyHostToDevice, st));
  HTAM_CK(cudaMemcpyAsync(kgroups, h_kg.data(), sizeof(KeyGroup) * h_kg.size(), cudaMemcpyHostToDevice, st));

  // 3. Stable slot assignment: pos[e] = old count of its group + rank among
  //    earlier rows of the batch with the same group.
  HTAM_CK(cudaMemsetAsync(hist, 0, sizeof(int32_t) * (size_t)G * n_chunks, st));
  chunk_hist_kernel<<<(unsigned)n_chunks, 256, 0, st>>>(gid, count, chunk, n_chunks, hist);
  HTAM_CK_LAUNCH("chunk_hist_kernel");
  chunk_scan_kernel<<<(unsigned)ceil_div((int64_t)G * 32, 256), 256, 0, st>>>(hist, n_chunks, G, m->count);
  HTAM_CK_LAUNCH("chunk_scan_kernel");
  chunk_place_kernel<<<(unsigned)ceil_div(n_chunks * 32, 256), 256, 0, st>>>(gid, count, chunk, n_chunks, hist, pos);
  HTAM_CK_LAUNCH("chunk_place_kernel");
  mark.launched(3);

  // 4. Copy rows into their slots.
  int vec_per_row = d * m->elem_bytes / 16;
  place_rows_kernel<<<(unsigned)ceil_div(count * 32, 256), 256, 0, st>>>(
      static_cast<const uint4 *>(entries), gid, pos, count, vec_per_row, m->page_list, m->page_off,
      static_cast<uint4 *>(m->pool), m->slot_id, m->n);
  HTAM_CK_LAUNCH("place_rows_kernel");
  mark.launched();

  // 5. Keys of the touched groups.
  if (!h_segs.empty()) {
    dim3 grid((unsigned)h_segs.size(), (unsigned)ceil_div(d, 256 * 8));
    if (m->dtype == HTAM_BF16) {
      key_partial_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(
          static_cast<const __nv_bfloat16 *>(m->pool), d, m->page_list, m->page_off, segs, partial);
    } else {
      key_partial_kernel<float><<<grid, 256, 0, st>>>(static_cast<const float *>(m->pool), d,
                                                      m->page_list, m->page_off, segs, partial);
    }
    HTAM_CK_LAUNCH("key_partial_kernel");
    dim3 g2((unsigned)h_kg.size(), (unsigned)std::min<int64_t>(ceil_div(d, 256), 16));
    key_finalize_kernel<<<g2, 256, 0, st>>>(kgroups, partial, d, m->csum, m->cent, m->cent_hi, m->cent_lo);
    HTAM_CK_LAUNCH("key_finalize_kernel");
    mark.launched(2);
  }

  // 6. New device counts and host mirrors.
  std::vector<int32_t> h_c32(G);
  for (int32_t g = 0; g < G; ++g) h_c32[g] = (int32_t)new_count[g];
  HTAM_CK(cudaMemcpyAsync(m->count, h_c32.data(), sizeof(int32_t) * G, cudaMemcpyHostToDevice, st));
  mark.end();
  // The host vectors above are pageable, so cudaMemcpyAsync staged them
  // before returning; the key and segment tables in scratch are read by the
  // kernels above in stream order, before any later call on the stream can
  // reuse the scratch (a reallocation frees it only after a device
  // synchronisation).  Nothing here needs to wait for the GPU.
  m->h_count.swap(new_count);
  m->n_pages_used = next_page;
  m->n += count;
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
  m->h_pages.assign(n_groups, {});

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
      cudaMalloc(&m->count, sizeof(int32_t) * n_groups) != cudaSuccess ||
      cudaMalloc(&m->csum, sizeof(double) * gd) != cudaSuccess ||
      cudaMalloc(&m->cent, sizeof(float) * gd) != cudaSuccess ||
      cudaMalloc(&m->cent_hi, sizeof(__nv_bfloat16) * gd) != cudaSuccess ||
      cudaMalloc(&m->cent_lo, sizeof(__nv_bfloat16) * gd) != cudaSuccess ||
      cudaMalloc(&m->status, sizeof(unsigned int)) != cudaSuccess) {
    cudaGetLastError();
    return fail(HTAM_ENOMEM);
  }
  // Empty rows are zero (never NaN), empty slots have id -1, keys start at 0.
  if (cudaMemsetAsync(m->pool, 0, pool_bytes, st) != cudaSuccess ||
      cudaMemsetAsync(m->slot_id, 0xff, sizeof(int32_t) * m->n_pages_max * kPageRows, st) != cudaSuccess ||
      cudaMemsetAsync(m->page_off, 0, sizeof(int32_t) * (n_groups + 1), st) != cudaSuccess ||
      cudaMemsetAsync(m->count, 0, sizeof(int32_t) * n_groups, st) != cudaSuccess ||
      cudaMemsetAsync(m->csum, 0, sizeof(double) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->cent, 0, sizeof(float) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->cent_hi, 0, sizeof(__nv_bfloat16) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->cent_lo, 0, sizeof(__nv_bfloat16) * gd, st) != cudaSuccess ||
      cudaMemsetAsync(m->status, 0, sizeof(unsigned int), st) != cudaSuccess) {
    set_last_error("cudaMemsetAsync", cudaGetLastError());
    return fail(HTAM_ECUDA);
  }
  htam_status s = add_rows(m, entries, gid, n, nullptr, st);
  if (s != HTAM_OK) return fail(s);
  *out = m;
  return HTAM_OK;
}

htam_status append_impl(htam_memory *m, const void *entries, const int32_t *gid, int64_t count,
                        int32_t *assigned, cudaStream_t st) {
  if (m->n + count > m->capacity) return HTAM_ECAPACITY;
  return add_rows(m, entries, gid, count, assigned, st);
}

}  // namespace htam
