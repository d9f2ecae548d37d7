/*
 * htam.h -- C ABI of the GB300 hierarchical transition-attended memory lookup
 * (HTAM, arxiv 2605.29734).
 *
 * The memory follows the paper's Hierarchical Transition Graph (Eq. 6, §4.1):
 * coarse *groups* stand for the global nodes V_G, fine *entries* (transition
 * embeddings) stand for the local nodes V_GL, and every entry has one parent
 * group (par(l) in Eq. 12).  Each group's key is the mean of its entries.
 *
 * A query runs the read side of one evolution step (§4.3, Algorithm 1 steps 2
 * and 3) for a batch of state embeddings q:
 *   1. score every non-empty group key with the linear scorer (Eq. 9 with
 *      phi = w^T z of App. B.6; in embedding space the dot product q . c_g)
 *      and keep the k_groups best groups (ties to the lower group id);
 *   2. restrict the candidates to the entries of the selected groups (Eq. 12),
 *      score them (q . k_e) and return the k_entries best (Eq. 13 as a top-k,
 *      ties to the lower entry id), with
 *      lse = log sum_{e in C} exp(s_e / tau) over the WHOLE candidate set C
 *      and weight w_e = eps/|C| + (1 - eps) * exp(s_e / tau - lse)
 *      (the eps-uniform / tau-softmax mixture of Eq. 11).
 * Appending entries is the memory update of Eq. 15: rows are filed under
 * their groups and the group keys are updated in place.
 *
 * Conventions for every function below:
 *  - Array pointers are DEVICE pointers (except in htam_query_host and the
 *    host-output helpers), row-major and contiguous, 16-byte aligned.
 *  - Entry and query rows are of the memory's dtype (fp32 or bf16).
 *  - Entry ids are the caller's numbering: the rows passed to
 *    htam_build_memory are ids 0..n-1, appended rows continue from the current
 *    entry count.  Ids are int32, so the capacity is below 2^31.
 *  - Work is queued on `cuda_stream` (a cudaStream_t; NULL = legacy default
 *    stream).  Inputs must stay valid until the queued work has finished;
 *    the library copies entries into its own storage.
 *  - Functions return a status and never abort or throw.  Argument errors are
 *    detected before anything is launched and leave the memory unchanged.
 *    The one check made on the device is that of an append's group ids (see
 *    htam_append_transitions): a rejected batch leaves the memory unchanged
 *    and is reported by htam_device_status.
 *  - One memory object is used from one stream at a time: htam_query does
 *    not modify the stored entries or keys, but it uses scratch space owned by
 *    the memory object, so two queries on the same object must not overlap.
 */
#ifndef HTAM_H_
#define HTAM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct htam_memory htam_memory; /* opaque, owns all its device storage */

typedef enum {
  HTAM_OK = 0,
  HTAM_EINVAL = 1,    /* bad argument (null, misaligned, out of range) */
  HTAM_ENOMEM = 2,    /* device or host allocation failed */
  HTAM_ECAPACITY = 3, /* append would exceed the memory's capacity */
  HTAM_ECUDA = 4,     /* a CUDA call or kernel launch failed */
  HTAM_ETIMEOUT = 5,  /* a bounded device-side wait gave up (kernel returned early) */
  HTAM_ENODEV = 6     /* no usable CUDA device */
} htam_status;

typedef enum { HTAM_F32 = 0, HTAM_BF16 = 1 } htam_dtype;

/* Query parameters.
 *  k_groups : groups kept per query, 1 <= k_groups <= min(n_groups, 64)
 *  k_entries: entries returned per query, 1 <= k_entries <= 64
 *  tau      : softmax temperature of Eq. 11, tau > 0 (the paper gives no
 *             value; 1 is the neutral choice)
 *  epsilon  : uniform-exploration mass of Eq. 11, 0 <= epsilon <= 1 */
typedef struct {
  int32_t k_groups;
  int32_t k_entries;
  float tau;
  float epsilon;
} htam_query_params;

/* Builds a memory from n entries (the initial memory M_0 of Algorithm 1).
 *  entries  : [n, d] of dtype, device
 *  group_ids: [n] int32 in [0, n_groups), device
 *  d        : embedding dimension, multiple of 8, 8 <= d <= 16384
 *  n_groups : number of groups, 1 <= n_groups <= 65536
 *  capacity : most entries the memory will ever hold (>= n, < 2^31); storage
 *             is reserved up front so that appends never reallocate
 *  out      : receives the new memory (NULL on failure)
 * The rows are laid out on the device as an append lays them out; the call
 * then synchronises `cuda_stream` once to read the group-id check, so a
 * build with a group id outside [0, n_groups) fails with EINVAL.  Errors:
 * EINVAL (arguments, a group id out of range), ENOMEM, ECUDA, ENODEV. */
htam_status htam_build_memory(const void *entries, const int32_t *group_ids,
                              int64_t n, int32_t d, int32_t n_groups,
                              htam_dtype dtype, int64_t capacity,
                              void *cuda_stream, htam_memory **out);

/* Appends `count` entries (the memory update of Eq. 15) and updates the keys
 * of the groups they join in place.  New entries get ids n, n+1, ... where n
 * counts the entries of every batch accepted before this one.
 *  entries  : [count, d] of the memory's dtype, device, 16-byte aligned
 *  group_ids: [count] int32, device, 16-byte aligned: a group in
 *             [0, n_groups), or -1 for an entry without a group, which joins
 *             the group whose key scores highest against it (q . c_g with the
 *             entry as q, stage 1's scorer; ties to the lower id; empty groups
 *             excluded), by the keys as they stand before this call
 * Fully asynchronous: the batch's group sizes, the nearest-key choices, the
 * page layout and the key updates are all computed on the device, with no
 * host round trip and no memset or copy in the stream (a growth of the
 * memory object's scratch or batch counters, on the first append of a new
 * size, synchronises the device once).  Page space never
 * runs out: the pages reserved at build hold any `capacity` entries.
 * The group ids are checked on the device.  A batch with an id out of range,
 * or an id of -1 while every group is empty, is rejected there: the memory
 * is left unchanged (no entry, key, size or id number is used up) and the
 * next htam_device_status call returns EINVAL.  Later calls queued behind a
 * rejected batch see the memory as it was.
 * Errors returned by the call itself: EINVAL (arguments), ECAPACITY (n +
 * count would exceed the capacity; appends the device rejected are
 * subtracted first), ENOMEM, ECUDA; the memory is unchanged on any of them. */
htam_status htam_append_transitions(htam_memory *m, const void *entries,
                                    const int32_t *group_ids, int64_t count,
                                    void *cuda_stream);

/* htam_append_transitions that also reports the group each entry joined:
 *  assigned : [count] int32, device, caller-allocated (may be group_ids
 *             itself); receives group_ids with every -1 replaced by the group
 *             chosen for that entry (left as it was if the device rejects the
 *             batch).
 * The nearest-key choice keeps a [rows, n_groups] fp32 score buffer that the
 * memory object owns (up to 16 MiB per K split), grown with cudaMalloc on
 * demand; its kernels are queued with every append and do nothing when no id
 * is -1. */
htam_status htam_append_assign(htam_memory *m, const void *entries,
                               const int32_t *group_ids, int64_t count,
                               int32_t *assigned, void *cuda_stream);

/* Answers b queries (device pointers; all outputs caller-allocated):
 *  queries     : [b, d] of the memory's dtype
 *  group_idx   : [b, k_groups] int32, selected groups best first, -1 padding
 *                when fewer than k_groups groups are non-empty
 *  group_score : [b, k_groups] fp32, q . c_g (-inf for padding)
 *  entry_idx   : [b, k_entries] int32 entry ids best first, -1 padding when
 *                the candidate set holds fewer than k_entries entries
 *  entry_score : [b, k_entries] fp32, q . k_e (-inf for padding)
 *  entry_weight: [b, k_entries] fp32, w_e as above (0 for padding)
 *  lse         : [b] fp32 or NULL, log-sum-exp of s/tau over the candidates
 * Fully asynchronous: nothing is read back.  0 <= b <= 2^24 (b may be 0).  A
 * device-side timeout is reported by htam_device_status.  Errors: EINVAL,
 * ENOMEM (scratch growth), ECUDA. */
htam_status htam_query(htam_memory *m, const void *queries, int32_t b,
                       const htam_query_params *p, int32_t *group_idx,
                       float *group_score, int32_t *entry_idx,
                       float *entry_score, float *entry_weight, float *lse,
                       void *cuda_stream);

/* The same lookup with every array in HOST memory (pageable or pinned): the
 * queries are copied to the device, htam_query runs, and the outputs are
 * copied back; returns after the stream has finished.  lse may be NULL. */
htam_status htam_query_host(htam_memory *m, const void *queries, int32_t b,
                            const htam_query_params *p, int32_t *group_idx,
                            float *group_score, int32_t *entry_idx,
                            float *entry_score, float *entry_weight,
                            float *lse, void *cuda_stream);

/* Longest prefix htam_query_prefix takes. */
#define HTAM_MAX_PREFIX 64

/* Prefix-attended lookup.  The global-direction score of Eq. 9 sums the
 * transition utility over the prefix of earlier directions (Eq. 8) with the
 * position-aware weights of Eq. 10:
 *   score(g) = sum_{i=1..P} alpha_i (q_i . c_g),  alpha_i = exp(-lambda (P - i)),
 * for a prefix q_1..q_P of state embeddings per query, q_P the most recent.
 * The scorer is linear in the query, so the call forms the reduced query
 * qbar = sum_i alpha_i q_i on the device (fp32 accumulation over i = 1..P,
 * rounded once to the memory's dtype) and runs the htam_query lookup on it:
 * both levels score qbar.
 *  prefix : [b, p_len, d] of the memory's dtype, device, 16-byte aligned
 *  p_len  : 1 <= p_len <= HTAM_MAX_PREFIX (p_len = 1 is htam_query itself)
 *  lambda : >= 0 and finite (the paper gives no value)
 * Outputs, asynchrony and errors as htam_query.  The reduced queries are kept
 * in a buffer the memory object owns, grown with cudaMalloc on demand. */
htam_status htam_query_prefix(htam_memory *m, const void *prefix, int32_t b, int32_t p_len,
                              float lambda, const htam_query_params *p, int32_t *group_idx,
                              float *group_score, int32_t *entry_idx, float *entry_score,
                              float *entry_weight, float *lse, void *cuda_stream);

/* Most features per edge htam_query_edges takes. */
#define HTAM_MAX_EDGE_FEATURES 32

/* Lookup routed by transition edges: the global router of Eq. 9 with the
 * transition utility of App. B.6, a fixed linear reward over the features of
 * the edge between two directions, phi(g_i, g) = w . z(g_i, g), summed over a
 * prefix of earlier directions with the weights of Eq. 10:
 *   score(g) = sum_{i=1..P} alpha_i w . Z[p_i][g][:],  alpha_i = exp(-lambda (P - i)).
 * These scores replace the group-key scores of stage 1 (the top k_groups
 * groups by score, ties to the lower id, empty groups never chosen,
 * group_score = these scores); stage 2 scores the selected groups' entries
 * against `queries` as htam_query does.
 *  edge_features : [n_groups, n_groups, n_features] fp32, device, 16-byte
 *                  aligned, row = from, column = to (caller-owned)
 *  n_features    : 1 <= n_features <= HTAM_MAX_EDGE_FEATURES (12 in App. B.6)
 *  weights       : [n_features] fp32, HOST, finite
 *  prefix_groups : [b, p_len] int32, HOST, group ids in [0, n_groups) or -1
 *                  for no element (contributes nothing); the most recent last
 *  p_len, lambda : as htam_query_prefix
 *  queries       : [b, d] of the memory's dtype, device (the stage-2 states)
 * Outputs, asynchrony and errors as htam_query (EINVAL also for a prefix id
 * out of range); the prefix is copied to the device inside the call. */
htam_status htam_query_edges(htam_memory *m, const float *edge_features, int32_t n_features,
                             const float *weights, const int32_t *prefix_groups, int32_t p_len,
                             float lambda, const void *queries, int32_t b,
                             const htam_query_params *p, int32_t *group_idx, float *group_score,
                             int32_t *entry_idx, float *entry_score, float *entry_weight,
                             float *lse, void *cuda_stream);

/* Seed and counter offset of the policy draws below.  The draws of query i
 * of a batch depend only on (seed, offset, i, group); pass a new offset (a
 * step counter, say) for fresh draws. */
typedef struct {
  uint64_t seed;
  uint64_t offset;
} htam_sampling;

/* Lookup with the groups DRAWN from the global-direction policy instead of
 * ranked (Algorithm 1, step 2: g_t ~ mu_g of Eq. 11):
 *   mu_g = epsilon / |G_t| + (1 - epsilon) * softmax(s_g / tau) over the
 *   non-empty groups G_t, s_g = q . c_g, tau and epsilon from `p`.
 * k_groups draws without replacement (k_groups = 1 is the paper's single
 * draw): the groups with the k_groups largest keys log mu_g - log(-log u_g)
 * (the Gumbel-top-k construction, Kool, van Hoof and Welling, ICML 2019),
 * ties to the lower id.  u_g is the query's uniform for group g: word (g mod 4)
 * of Philox4x32-10 (Salmon et al., SC 2011) at counter (g / 4, i, low and high
 * words of offset) under key (low and high words of seed), its top 23 bits
 * plus one half times 2^-23.  group_idx lists the draws in order and
 * group_score holds their scores q . c_g; stage 2 and every other output are
 * those of htam_query over the drawn groups.  Arguments and errors as
 * htam_query (EINVAL also for sampling == NULL); the call waits for the group
 * sizes of the last queued append (the policy's |G_t| is the exact number of
 * non-empty groups), otherwise it is asynchronous. */
htam_status htam_query_sampled(htam_memory *m, const void *queries, int32_t b,
                               const htam_query_params *p, const htam_sampling *sampling,
                               int32_t *group_idx, float *group_score, int32_t *entry_idx,
                               float *entry_score, float *entry_weight, float *lse,
                               void *cuda_stream);

/* htam_query_edges with the groups drawn from the policy of Eq. 11 over the
 * edge-table scores of Eq. 9, as htam_query_sampled draws them (the paper's
 * global direction choice as Algorithm 1 states it). */
htam_status htam_query_edges_sampled(htam_memory *m, const float *edge_features, int32_t n_features,
                                     const float *weights, const int32_t *prefix_groups, int32_t p_len,
                                     float lambda, const void *queries, int32_t b,
                                     const htam_query_params *p, const htam_sampling *sampling,
                                     int32_t *group_idx, float *group_score, int32_t *entry_idx,
                                     float *entry_score, float *entry_weight, float *lse,
                                     void *cuda_stream);

/* Flat scan: stage 2 of the lookup with every entry a candidate, no group
 * stage.  This is the flat memory retrieval the paper compares against
 * (App. C.4, and the "w/o hierarchy" ablation of App. C.8); its result equals
 * htam_query with k_groups = the number of non-empty groups.  The fine scores
 * s = q . k_e over all n entries, the softmax of Eq. 11 over all of them
 * (|C| = n in the epsilon term), and the k_entries best by Eq. 13 (ties to the
 * lower id).
 *  queries     : [b, d] of the memory's dtype, device, 16-byte aligned
 *  k_entries   : 1 <= k_entries <= 64
 *  tau, epsilon: as htam_query_params
 *  entry_idx / entry_score / entry_weight / lse: as htam_query ([b, k_entries],
 *                lse [b] or NULL), -1 / -inf / 0 padding when n < k_entries
 * 0 <= b <= 2^24 and b * (non-empty groups) <= 2^28.  Outputs and errors as
 * htam_query; the call waits for the group sizes of the last queued append
 * (it needs the exact non-empty groups), otherwise it is asynchronous. */
htam_status htam_query_flat(htam_memory *m, const void *queries, int32_t b,
                            int32_t k_entries, float tau, float epsilon,
                            int32_t *entry_idx, float *entry_score,
                            float *entry_weight, float *lse, void *cuda_stream);

/* Bytes of the fixed device scratch used by htam_select_groups_static. */
#define HTAM_STATIC_SCRATCH_BYTES (16u << 20)

/* Group selection that allocates nothing.  The paper has no counterpart: this
 * is an extra entry point for callers that cannot allocate device memory
 * while they run -- a server whose device memory is fully reserved up front
 * (an allocation could fail or fragment its pool), code running inside an
 * allocator callback that must not re-enter the allocator, and latency-
 * critical loops that cannot absorb the device-wide synchronisation that
 * cudaFree implies.  htam_query may grow the memory object's scratch with
 * cudaMalloc; this call never calls cudaMalloc, cudaFree or any allocating
 * library routine.
 *
 * It returns the group_idx / group_score of htam_query's stage 1 (the coarse
 * scores q . c_g against every non-empty group key and the k_groups best
 * groups, ties to the lower id, -1 / -inf padding), with scores equal within
 * fp32 rounding (so groups whose scores differ by less than that may come
 * out in the other order).  Arguments are those
 * of htam_query: device pointers, queries [b, d] of the memory's dtype,
 * outputs [b, k_groups], 0 <= b <= 2^24.
 *
 * Scratch: the [b, n_groups] fp32 score matrix lives in one fixed array of
 * HTAM_STATIC_SCRATCH_BYTES compiled into the library; every GPU that loads
 * the library keeps it until the process exits.  Calls with
 * b * n_groups * 4 > HTAM_STATIC_SCRATCH_BYTES are rejected with HTAM_EINVAL
 * before anything is launched.  The first call on a device looks up the
 * array's device address (cudaGetSymbolAddress, with that device current);
 * make that first call before any stream capture.  The current device must be
 * the memory's device.  All calls share the array and it keeps the previous
 * call's contents (each call writes what it reads, so nothing needs to start
 * at zero); calls whose GPU work overlaps -- on different streams or from
 * different host threads -- race on it and must be serialised by the caller.
 * Errors: EINVAL, ECUDA. */
htam_status htam_select_groups_static(const htam_memory *m, const void *queries,
                                      int32_t b, int32_t k_groups,
                                      int32_t *group_idx, float *group_score,
                                      void *cuda_stream);

/* Sizes of a memory; any output pointer may be NULL (host pointers).  *n
 * waits for the last queued append to finish (and excludes any batch the
 * device rejected). */
htam_status htam_memory_info(const htam_memory *m, int64_t *n, int32_t *d,
                             int32_t *n_groups, int64_t *capacity);

/* Copies the current group sizes n_g into counts[n_groups] (host), after
 * waiting for the last queued append to finish. */
htam_status htam_memory_group_counts(const htam_memory *m, int64_t *counts);

/* Copies the current group keys (fp32 means, [n_groups, d]) into host
 * memory; rows of empty groups are zero.  Synchronises `cuda_stream`. */
htam_status htam_memory_group_keys(const htam_memory *m, float *keys,
                                   void *cuda_stream);

/* Synchronises `cuda_stream`, reads and clears the memory's device status
 * word.  Returns ETIMEOUT if a bounded device wait gave up since the last
 * check, else EINVAL if the device rejected an append's group ids since the
 * last check (see htam_append_transitions), ECUDA if the stream reports an
 * error, OK otherwise. */
htam_status htam_device_status(htam_memory *m, void *cuda_stream);

/* Phases of htam_query (and of htam_append_transitions), for the timing
 * counters below. */
typedef enum {
  HTAM_PHASE_COARSE = 0, /* group-key scores */
  HTAM_PHASE_SELECT = 1, /* top-k_groups per query */
  HTAM_PHASE_BUCKET = 2, /* group -> queries buckets and work units */
  HTAM_PHASE_FINE = 3,    /* entry scores of small buckets on the CUDA cores */
  HTAM_PHASE_FINE_TC = 4, /* entry scores of large buckets on the tensor cores */
  HTAM_PHASE_MERGE = 5,   /* per-query merge, weights, outputs */
  HTAM_PHASE_PREFIX = 6,  /* reduced queries of htam_query_prefix */
  HTAM_PHASE_APPEND = 7,  /* htam_append_transitions / htam_append_assign, from the
                             batch's group count to the last key update */
  HTAM_N_PHASES = 8
} htam_phase;

/* Tuning knobs of htam_query (all paths return the same results within the
 * fp32 rounding of the scores):
 *  HTAM_TUNE_TC_MIN_BUCKET: when a group was selected by at least this many
 *    queries of a batch, its entries are scored against them on the tensor
 *    cores (tcgen05, 128 queries per tile); smaller buckets are scored on the
 *    CUDA cores.  Needs a bf16 memory and k_entries <= 32.  Default 2 (a
 *    bucket of one query is matrix-vector work, streamed on the CUDA cores);
 *    a value above the batch size turns the tensor-core path off.  >= 1.
 *  HTAM_TUNE_STREAM_ROWS: 1 (default) prefetches the CUDA-core path's entry
 *    rows into per-warp shared-memory rings (bf16 memories with rows up to
 *    8 KiB and k_entries <= 32); 0 loads them directly into registers.
 *  HTAM_TUNE_TC_PAIRS: 1 scores the tensor-core buckets of more than 128
 *    queries on pairs of SMs (two 128-query chunks per M=256 MMA,
 *    cta_group::2, each SM staging half of every entry tile); 0 (default)
 *    runs every chunk on one SM.
 *  HTAM_TUNE_PDL: 1 (default) launches the kernels of a query or an append
 *    with programmatic stream serialisation, so that each kernel's blocks
 *    are scheduled while the previous kernel finishes (every such kernel
 *    waits for its predecessor before touching memory); 0 launches them
 *    plainly.  The results are the same either way.
 *  HTAM_TUNE_FINE_OVERLAP: 1 (default) runs the CUDA-core and tensor-core
 *    fine kernels of a query concurrently: the CUDA-core kernel goes to an
 *    internal stream of the memory object, forked from `cuda_stream` and
 *    joined back to it by events inside the call (so the call still orders
 *    as one unit of work on `cuda_stream`, and stream capture records the
 *    fork and join); 0 runs them one after the other on `cuda_stream`.
 * Errors: EINVAL (m NULL, unknown key, value out of range). */
typedef enum {
  HTAM_TUNE_TC_MIN_BUCKET = 0,
  HTAM_TUNE_STREAM_ROWS = 1,
  HTAM_TUNE_TC_PAIRS = 2,
  HTAM_TUNE_PDL = 3,
  HTAM_TUNE_FINE_OVERLAP = 4
} htam_tuning;
htam_status htam_set_tuning(htam_memory *m, htam_tuning key, int32_t value);

/* Reads a tuning value (the keys and defaults of htam_set_tuning) into
 * *value.  Errors: EINVAL (m or value NULL, unknown key). */
htam_status htam_get_tuning(const htam_memory *m, htam_tuning key, int32_t *value);

/* Turns CUDA-event timing of each htam_query phase (and of each append) on
 * (1) or off (0).  While on, every call records a pair of events around each
 * phase on its stream (a few microseconds of host work per call). */
htam_status htam_set_phase_timing(htam_memory *m, int enable);

/* Synchronises `cuda_stream`, then writes, for the htam_query calls since the
 * previous read: ms[p] = summed device time of phase p (0 unless timing was
 * on), launches[p] = kernels phase p launched, *queries = calls.  Any output
 * may be NULL; arrays hold HTAM_N_PHASES values (host).  Resets the counts. */
htam_status htam_read_phase_timing(htam_memory *m, double *ms, int64_t *launches,
                                   int64_t *queries, void *cuda_stream);

/* Releases the memory and all its device storage (NULL is a no-op).  The
 * caller must make sure no queued work still uses it. */
void htam_free_memory(htam_memory *m);

/* Human-readable name of a status code (static string). */
const char *htam_status_string(htam_status s);

/* Text of the last failing CUDA call made by this thread ("" if none); the
 * string stays valid until the thread's next failing call. */
const char *htam_last_error(void);

/* Diagnostic for the bounded-wait machinery: launches one kernel that waits
 * for a device flag that nothing sets, giving up after `max_iters` polls; the
 * kernel records the give-up in a status word and returns.  Returns ETIMEOUT
 * when the wait gave up (the expected result), OK if it did not, ECUDA on a
 * launch error.  Synchronises `cuda_stream`.  The paper has no counterpart;
 * it exists to test failure reporting without faulting the GPU. */
htam_status htam_selftest_wait_timeout(int64_t max_iters, void *cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* HTAM_H_ */
