// internal.h -- the memory object behind the opaque htam_memory handle.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "htam.h"

struct htam_memory {
  int device = 0;
  int sm_count = 0;
  int32_t d = 0;
  int32_t n_groups = 0;
  htam_dtype dtype = HTAM_BF16;
  int elem_bytes = 2;
  // Entries stored, as the host sees it: the device's count at the last
  // adopted mirror plus the rows of every append queued since (an append the
  // device rejects is subtracted once a later mirror shows it).
  int64_t n = 0;
  int64_t capacity = 0;    // most entries ever stored
  int64_t n_pages_max = 0; // pages reserved: ceil(capacity/128) + n_groups

  // Paged storage: page p holds rows [p*128, p*128+128) of `pool`; each row
  // is d elements of dtype.  Group g owns pages page_list[page_off[g] ..
  // page_off[g+1]) in order, filled front to back; its i-th entry sits in
  // page page_list[page_off[g] + i/128], row i%128.
  void *pool = nullptr;
  int32_t *slot_id = nullptr;    // [n_pages_max*128] entry id of each row, -1 if empty
  int32_t *page_list = nullptr;  // [n_pages_max]
  int32_t *page_off = nullptr;   // [n_groups+1]
  // The layout an append writes (it reads the one above); the host swaps the
  // two pairs after queueing each append, so the pair above is always the
  // current one in stream order.
  int32_t *page_list_alt = nullptr;
  int32_t *page_off_alt = nullptr;
  int32_t *count = nullptr;      // [n_groups] entries per group (device copy)
  int64_t *dev_ctr = nullptr;    // [2] entries stored, pages used (device)

  // Group keys: fp64 running sums (exact enough to update in place), the
  // fp32 mean, and the mean split into bf16 hi + lo parts.
  double *csum = nullptr;           // [n_groups*d]
  float *cent = nullptr;            // [n_groups*d]
  __nv_bfloat16 *cent_hi = nullptr; // [n_groups*d]
  __nv_bfloat16 *cent_lo = nullptr; // [n_groups*d]

  unsigned int *status = nullptr;   // device status word (bit 0: a wait gave up)

  // Host mirror of the group sizes, exact as of the append numbered
  // mirror_seq; rows_pending rows were queued after it.  Appends run on the
  // device without a host round trip: in each one the key finalisation
  // kernel writes the device sizes and entry count into a slot of a small
  // ring of mapped pinned memory, and an event is recorded after it; a later
  // call adopts the newest slot whose event has completed
  // (htam_device_status and the introspection calls wait for it).
  static constexpr int kMirrorSlots = 4;
  std::vector<int64_t> h_count;
  int64_t rows_pending = 0;
  int64_t rows_issued = 0;       // rows of all appends queued (and the build)
  int64_t append_seq = 0;        // appends queued
  int64_t mirror_seq = 0;        // the append the mirror reflects
  void *h_pin = nullptr;         // kMirrorSlots x (int64 n, int32 counts[G])
  void *d_pin = nullptr;         // h_pin as the device sees it (the last append kernel writes the slots)
  int32_t *batch_ctr = nullptr;  // batch counters of add_rows, zero between batches
  int64_t batch_ctr_len = 0;
  bool batch_dirty = false;       // a batch stopped before clearing them
  uint32_t *qbits = nullptr;      // bucket bitmap of the multi-kernel bucketing, zero between queries
  int64_t qbits_len = 0;
  bool qbits_dirty = false;       // a query stopped before clearing it
  size_t pin_slot_bytes = 0;
  cudaEvent_t mirror_ev[kMirrorSlots] = {};
  int64_t slot_seq[kMirrorSlots] = {};       // append number each slot holds (0 = none)
  int64_t slot_rows_issued[kMirrorSlots] = {};
  cudaStream_t last_stream = nullptr;        // stream of the last append

  // Scratch owned by the object, grown on demand (never shrinks).
  void *scratch = nullptr;
  size_t scratch_bytes = 0;
  // Device staging for htam_query_host.
  void *stage = nullptr;
  size_t stage_bytes = 0;
  // Reduced queries of htam_query_prefix.
  void *prefix_buf = nullptr;
  size_t prefix_bytes = 0;
  void *assign_buf = nullptr;  // nearest-key assignment of appended rows
  size_t assign_bytes = 0;

  // Phase timing and launch counters (htam_set_phase_timing / _read_).
  bool timing = false;
  std::vector<cudaEvent_t> ev_pool;    // created on demand, reused
  std::vector<int> ev_phase;           // phase of each recorded pair
  size_t ev_used = 0;                  // events in use (2 per pair)
  int64_t n_queries = 0;
  int64_t phase_launches[HTAM_N_PHASES] = {};

  // Tensor-core fine path: smallest bucket it takes (set at build from d),
  // and the TMA map of the page pool (built on first use).
  int tc_min = 16;
  // CUDA-core fine path: stream rows through shared memory (1) or load them
  // directly (0).
  int stream_rows = 1;
  // Tensor-core buckets of more than one 128-query chunk on SM pairs (1) or
  // single SMs (0).  Off by default: the epilogue, not the operand feed,
  // limits the kernel, and the pair path measured slower.
  int tc_pairs = 0;
  // Kernels of a query or append launched with programmatic stream
  // serialisation (1, default) or as plain launches (0).
  int pdl = 1;
  // The CUDA-core and tensor-core fine kernels of a query run concurrently
  // (1: the CUDA-core kernel on an internal stream forked from and joined
  // back to the caller's by events) or one after the other (0).
  int fine_overlap = 1;
  cudaStream_t side = nullptr;   // created on first use
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  CUtensorMap pool_map;
  bool pool_map_ready = false;
};

namespace htam {

// Grows m->scratch to at least `bytes` (synchronising the device when it has
// to reallocate).  Returns HTAM_OK / HTAM_ENOMEM.
htam_status ensure_scratch(htam_memory *m, size_t bytes);

// Bump allocator over a scratch buffer (256-byte aligned pieces).
struct Carver {
  char *base;
  size_t off = 0;
  explicit Carver(void *b) : base(static_cast<char *>(b)) {}
  template <typename T>
  T *take(size_t count) {
    off = (off + 255) & ~size_t(255);
    T *p = reinterpret_cast<T *>(base + off);
    off += count * sizeof(T);
    return p;
  }
  static size_t round(size_t bytes) { return (bytes + 255) & ~size_t(255); }
};

// Adopts the newest completed mirror slot.  wait = true first waits for the
// newest slot's event (the mirror is then exact unless a later append was
// queued meanwhile).  Returns HTAM_ECUDA if waiting failed.
htam_status refresh_mirror(htam_memory *m, bool wait);

htam_status build_impl(const void *entries, const int32_t *group_ids, int64_t n, int32_t d,
                       int32_t n_groups, htam_dtype dtype, int64_t capacity, cudaStream_t st,
                       htam_memory **out);
htam_status append_impl(htam_memory *m, const void *entries, const int32_t *group_ids,
                        int64_t count, int32_t *assigned, cudaStream_t st);
// Stage 1 from a transition-edge table instead of the group keys
// (htam_query_edges).
struct EdgeRoute {
  const float *Z;          // [G, G, F] device, from x to x feature
  const int32_t *prefix;   // [B, P] host, ids in [-1, G)
  int F, P;
  float w[HTAM_MAX_EDGE_FEATURES];
  float alpha[HTAM_MAX_PREFIX];
};
// Seed and counter offset of the policy draws (Algorithm 1, step 2).
struct SampleSpec {
  uint64_t seed, offset;
};
htam_status query_impl(htam_memory *m, const void *queries, int32_t b,
                       const htam_query_params &p, int32_t *group_idx, float *group_score,
                       int32_t *entry_idx, float *entry_score, float *entry_weight, float *lse,
                       cudaStream_t st, const EdgeRoute *er = nullptr, bool flat = false,
                       const SampleSpec *smp = nullptr);
// Largest b * (non-empty groups) the flat scan takes (its bucket rows).
constexpr int64_t kMaxFlatRows = int64_t(1) << 28;
void free_impl(htam_memory *m);
// Rows of `entries` whose id in gid is -1 join the group whose key scores
// highest against them (stage 1's scorer and ranking with k = 1, by the keys
// as they stand before the append).  Queued without a host round trip: every
// kernel is gated on *n_unassigned (the batch's tally of such rows, on the
// device) and does nothing when it is zero.  For each such row e: ids[e] =
// the chosen group, bcount[that group] += 1 and hist[that group * n_chunks
// + e / chunk] += 1 (the stable sort's counts); a row that finds no
// non-empty group sets *bad.  Scratch: m->assign_buf, grown with cudaMalloc
// on demand (a growth synchronises the device).
struct PhaseMark;
htam_status assign_unassigned(htam_memory *m, const void *entries, const int32_t *gid, int64_t count,
                              const int32_t *n_unassigned, int32_t *ids, int32_t *bcount, int32_t *bad,
                              int32_t *hist, int64_t chunk, int64_t n_chunks, cudaStream_t st,
                              PhaseMark *mark = nullptr);

// Weights alpha_1..alpha_P of a prefix (Eq. 10), passed by value to the
// reduction kernel.
struct PrefixWeights {
  float alpha[HTAM_MAX_PREFIX];
};
// out[q] = sum_i alpha_i prefix[q][i] for b queries ([b, p_len, d] of the
// memory's dtype in, [b, d] out), fp32 accumulation, one rounding.
htam_status launch_prefix_reduce(const htam_memory *m, const void *prefix, int32_t b, int32_t p_len,
                                 const PrefixWeights &w, void *out, cudaStream_t st);

// Records the start / end of a query phase when timing is on, and counts
// kernel launches per phase.
struct PhaseMark {
  htam_memory *m;
  cudaStream_t st;
  int phase = -1;
  PhaseMark(htam_memory *mem, cudaStream_t s) : m(mem), st(s) {}
  // A phase begun but not ended (an error return) is dropped.
  ~PhaseMark() {
    if (m->timing && m->ev_phase.size() * 2 == m->ev_used + 2) m->ev_phase.pop_back();
  }
  void begin(int p);
  void end();
  void launched(int n = 1) { m->phase_launches[phase] += n; }
};

}  // namespace htam
