// api.cu -- the C ABI declared in include/htam.h: argument checks, status
// codes, and the bounded-wait self test.  Every argument error is detected
// here, before anything is launched.

#include <cmath>
#include <cstdio>
#include <cstring>

#include "common.cuh"
#include "internal.h"

namespace htam {

static thread_local char g_last_error[256] = "";
thread_local bool g_launch_pdl = false;

void set_last_error(const char *what, cudaError_t err) {
  std::snprintf(g_last_error, sizeof g_last_error, "%s: %s", what, cudaGetErrorString(err));
}

static bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Waits for a flag that nothing sets, giving up after max_iters polls; the
// give-up is recorded in *status and the kernel returns normally.
__global__ void wait_timeout_selftest_kernel(const volatile unsigned int *flag, long long max_iters,
                                             unsigned int *status) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  long long it = 0;
  while (*flag == 0u) {
    if (++it > max_iters) {
      atomicOr(status, 1u);
      return;
    }
    __nanosleep(64);
  }
}

void PhaseMark::begin(int p) {
  phase = p;
  if (!m->timing) return;
  while (m->ev_pool.size() < m->ev_used + 2) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) {
      cudaGetLastError();
      return;
    }
    m->ev_pool.push_back(e);
  }
  cudaEventRecord(m->ev_pool[m->ev_used], st);
  m->ev_phase.push_back(p);
}

void PhaseMark::end() {
  if (!m->timing || m->ev_phase.size() * 2 != m->ev_used + 2) return;
  cudaEventRecord(m->ev_pool[m->ev_used + 1], st);
  m->ev_used += 2;
}

}  // namespace htam

using namespace htam;

extern "C" {

const char *htam_status_string(htam_status s) {
  switch (s) {
    case HTAM_OK: return "HTAM_OK";
    case HTAM_EINVAL: return "HTAM_EINVAL: invalid argument";
    case HTAM_ENOMEM: return "HTAM_ENOMEM: allocation failed";
    case HTAM_ECAPACITY: return "HTAM_ECAPACITY: memory capacity exceeded";
    case HTAM_ECUDA: return "HTAM_ECUDA: CUDA error";
    case HTAM_ETIMEOUT: return "HTAM_ETIMEOUT: a device-side wait gave up";
    case HTAM_ENODEV: return "HTAM_ENODEV: no CUDA device";
  }
  return "unknown htam_status";
}

const char *htam_last_error(void) { return g_last_error; }

static htam_status check_device() {
  int n = 0;
  if (cudaGetDeviceCount(&n) != cudaSuccess || n == 0) {
    cudaGetLastError();
    return HTAM_ENODEV;
  }
  return HTAM_OK;
}

htam_status htam_build_memory(const void *entries, const int32_t *group_ids, int64_t n, int32_t d,
                              int32_t n_groups, htam_dtype dtype, int64_t capacity, void *cuda_stream,
                              htam_memory **out) {
  if (!out) return HTAM_EINVAL;
  *out = nullptr;
  if (dtype != HTAM_F32 && dtype != HTAM_BF16) return HTAM_EINVAL;
  if (d < 8 || d > 16384 || d % 8 != 0) return HTAM_EINVAL;
  if (n_groups < 1 || n_groups > 65536) return HTAM_EINVAL;
  if (n < 0 || capacity < n || capacity < 1 || capacity >= (int64_t(1) << 31) - kPageRows) return HTAM_EINVAL;
  if (n > 0 && (!entries || !group_ids || !aligned16(entries) || !aligned16(group_ids))) return HTAM_EINVAL;
  htam_status s = check_device();
  if (s != HTAM_OK) return s;
  return build_impl(entries, group_ids, n, d, n_groups, dtype, capacity,
                    static_cast<cudaStream_t>(cuda_stream), out);
}

htam_status htam_append_transitions(htam_memory *m, const void *entries, const int32_t *group_ids,
                                    int64_t count, void *cuda_stream) {
  if (!m || count < 0) return HTAM_EINVAL;
  if (count == 0) return HTAM_OK;
  if (!entries || !group_ids || !aligned16(entries) || !aligned16(group_ids)) return HTAM_EINVAL;
  return append_impl(m, entries, group_ids, count, nullptr, static_cast<cudaStream_t>(cuda_stream));
}

htam_status htam_append_assign(htam_memory *m, const void *entries, const int32_t *group_ids, int64_t count,
                               int32_t *assigned, void *cuda_stream) {
  if (!m || count < 0) return HTAM_EINVAL;
  if (count == 0) return HTAM_OK;
  if (!entries || !group_ids || !assigned || !aligned16(entries) || !aligned16(group_ids)) return HTAM_EINVAL;
  return append_impl(m, entries, group_ids, count, assigned, static_cast<cudaStream_t>(cuda_stream));
}

static htam_status check_query_args(const htam_memory *m, const void *queries, int32_t b,
                                    const htam_query_params *p, const int32_t *group_idx,
                                    const float *group_score, const int32_t *entry_idx,
                                    const float *entry_score, const float *entry_weight) {
  if (!m || !p || b < 0) return HTAM_EINVAL;
  if (p->k_groups < 1 || p->k_groups > kMaxK || p->k_groups > m->n_groups) return HTAM_EINVAL;
  if (p->k_entries < 1 || p->k_entries > kMaxK) return HTAM_EINVAL;
  if (!(p->tau > 0.0f) || !(p->epsilon >= 0.0f && p->epsilon <= 1.0f)) return HTAM_EINVAL;
  if (!std::isfinite(1.0f / p->tau)) return HTAM_EINVAL;
  if (b > (1 << 24)) return HTAM_EINVAL;
  if (b > 0 && (!queries || !group_idx || !group_score || !entry_idx || !entry_score || !entry_weight)) {
    return HTAM_EINVAL;
  }
  return HTAM_OK;
}

htam_status htam_query(htam_memory *m, const void *queries, int32_t b, const htam_query_params *p,
                       int32_t *group_idx, float *group_score, int32_t *entry_idx, float *entry_score,
                       float *entry_weight, float *lse, void *cuda_stream) {
  htam_status s = check_query_args(m, queries, b, p, group_idx, group_score, entry_idx, entry_score, entry_weight);
  if (s != HTAM_OK) return s;
  if (b > 0 && !aligned16(queries)) return HTAM_EINVAL;
  return query_impl(m, queries, b, *p, group_idx, group_score, entry_idx, entry_score, entry_weight, lse,
                    static_cast<cudaStream_t>(cuda_stream));
}

htam_status htam_query_prefix(htam_memory *m, const void *prefix, int32_t b, int32_t p_len, float lambda,
                              const htam_query_params *p, int32_t *group_idx, float *group_score,
                              int32_t *entry_idx, float *entry_score, float *entry_weight, float *lse,
                              void *cuda_stream) {
  htam_status s = check_query_args(m, prefix, b, p, group_idx, group_score, entry_idx, entry_score, entry_weight);
  if (s != HTAM_OK) return s;
  if (p_len < 1 || p_len > HTAM_MAX_PREFIX || !(lambda >= 0.f) || !std::isfinite(lambda)) return HTAM_EINVAL;
  if (b > 0 && !aligned16(prefix)) return HTAM_EINVAL;
  if (b == 0) return HTAM_OK;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const size_t bytes = (size_t)b * m->d * m->elem_bytes;
  if (bytes > m->prefix_bytes) {
    if (m->prefix_buf) cudaFree(m->prefix_buf);  // synchronises: no queued work still reads it
    m->prefix_buf = nullptr;
    m->prefix_bytes = 0;
    const size_t want = bytes + bytes / 2;
    if (cudaMalloc(&m->prefix_buf, want) != cudaSuccess) {
      cudaGetLastError();
      return HTAM_ENOMEM;
    }
    m->prefix_bytes = want;
  }
  PdlScope pdl(m->pdl != 0);
  PrefixWeights w;
  for (int i = 1; i <= p_len; ++i) w.alpha[i - 1] = (float)std::exp(-(double)lambda * (double)(p_len - i));
  PhaseMark mark(m, st);
  mark.begin(HTAM_PHASE_PREFIX);
  s = launch_prefix_reduce(m, prefix, b, p_len, w, m->prefix_buf, st);
  if (s != HTAM_OK) return s;
  mark.launched();
  mark.end();
  return query_impl(m, m->prefix_buf, b, *p, group_idx, group_score, entry_idx, entry_score, entry_weight, lse,
                    st);
}

htam_status htam_query_sampled(htam_memory *m, const void *queries, int32_t b, const htam_query_params *p,
                               const htam_sampling *sampling, int32_t *group_idx, float *group_score,
                               int32_t *entry_idx, float *entry_score, float *entry_weight, float *lse,
                               void *cuda_stream) {
  htam_status s = check_query_args(m, queries, b, p, group_idx, group_score, entry_idx, entry_score, entry_weight);
  if (s != HTAM_OK) return s;
  if (!sampling || (b > 0 && !aligned16(queries))) return HTAM_EINVAL;
  const SampleSpec smp{sampling->seed, sampling->offset};
  return query_impl(m, queries, b, *p, group_idx, group_score, entry_idx, entry_score, entry_weight, lse,
                    static_cast<cudaStream_t>(cuda_stream), nullptr, false, &smp);
}

static htam_status query_edges_impl(htam_memory *m, const float *edge_features, int32_t n_features,
                                    const float *weights, const int32_t *prefix_groups, int32_t p_len, float lambda,
                                    const void *queries, int32_t b, const htam_query_params *p, int32_t *group_idx,
                                    float *group_score, int32_t *entry_idx, float *entry_score,
                                    float *entry_weight, float *lse, void *cuda_stream, const SampleSpec *smp) {
  htam_status s = check_query_args(m, queries, b, p, group_idx, group_score, entry_idx, entry_score, entry_weight);
  if (s != HTAM_OK) return s;
  if (b > 0 && !aligned16(queries)) return HTAM_EINVAL;
  if (!edge_features || !aligned16(edge_features) || !weights || n_features < 1 ||
      n_features > HTAM_MAX_EDGE_FEATURES) {
    return HTAM_EINVAL;
  }
  if (p_len < 1 || p_len > HTAM_MAX_PREFIX || !(lambda >= 0.f) || !std::isfinite(lambda)) return HTAM_EINVAL;
  if (b > 0 && !prefix_groups) return HTAM_EINVAL;
  for (int f = 0; f < n_features; ++f) {
    if (!std::isfinite(weights[f])) return HTAM_EINVAL;
  }
  for (int64_t i = 0; i < (int64_t)b * p_len; ++i) {
    if (prefix_groups[i] < -1 || prefix_groups[i] >= m->n_groups) return HTAM_EINVAL;
  }
  if (b == 0) return HTAM_OK;
  EdgeRoute er;
  er.Z = edge_features;
  er.prefix = prefix_groups;
  er.F = n_features;
  er.P = p_len;
  for (int f = 0; f < HTAM_MAX_EDGE_FEATURES; ++f) er.w[f] = f < n_features ? weights[f] : 0.f;
  for (int i = 0; i < HTAM_MAX_PREFIX; ++i) {
    er.alpha[i] = i < p_len ? (float)std::exp(-(double)lambda * (double)(p_len - 1 - i)) : 0.f;
  }
  return query_impl(m, queries, b, *p, group_idx, group_score, entry_idx, entry_score, entry_weight, lse,
                    static_cast<cudaStream_t>(cuda_stream), &er, false, smp);
}

htam_status htam_query_edges(htam_memory *m, const float *edge_features, int32_t n_features, const float *weights,
                             const int32_t *prefix_groups, int32_t p_len, float lambda, const void *queries, int32_t b,
                             const htam_query_params *p, int32_t *group_idx, float *group_score, int32_t *entry_idx,
                             float *entry_score, float *entry_weight, float *lse, void *cuda_stream) {
  return query_edges_impl(m, edge_features, n_features, weights, prefix_groups, p_len, lambda, queries, b, p,
                          group_idx, group_score, entry_idx, entry_score, entry_weight, lse, cuda_stream, nullptr);
}

htam_status htam_query_edges_sampled(htam_memory *m, const float *edge_features, int32_t n_features,
                                     const float *weights, const int32_t *prefix_groups, int32_t p_len,
                                     float lambda, const void *queries, int32_t b, const htam_query_params *p,
                                     const htam_sampling *sampling, int32_t *group_idx, float *group_score,
                                     int32_t *entry_idx, float *entry_score, float *entry_weight, float *lse,
                                     void *cuda_stream) {
  if (!sampling) return HTAM_EINVAL;
  const SampleSpec smp{sampling->seed, sampling->offset};
  return query_edges_impl(m, edge_features, n_features, weights, prefix_groups, p_len, lambda, queries, b, p,
                          group_idx, group_score, entry_idx, entry_score, entry_weight, lse, cuda_stream, &smp);
}

htam_status htam_query_flat(htam_memory *m, const void *queries, int32_t b, int32_t k_entries, float tau,
                            float epsilon, int32_t *entry_idx, float *entry_score, float *entry_weight, float *lse,
                            void *cuda_stream) {
  if (!m || b < 0 || b > (1 << 24)) return HTAM_EINVAL;
  if (k_entries < 1 || k_entries > kMaxK) return HTAM_EINVAL;
  if (!(tau > 0.0f) || !(epsilon >= 0.0f && epsilon <= 1.0f) || !std::isfinite(1.0f / tau)) return HTAM_EINVAL;
  if (b > 0 && (!queries || !aligned16(queries) || !entry_idx || !entry_score || !entry_weight)) return HTAM_EINVAL;
  if (b == 0) return HTAM_OK;
  htam_status s = refresh_mirror(m, true);  // the exact non-empty groups (after any queued append)
  if (s != HTAM_OK) return s;
  int64_t nonempty = 0;
  for (int64_t c : m->h_count) nonempty += c > 0;
  if ((int64_t)b * std::max<int64_t>(1, nonempty) > kMaxFlatRows) return HTAM_EINVAL;
  const htam_query_params p{(int32_t)std::max<int64_t>(1, nonempty), k_entries, tau, epsilon};
  return query_impl(m, queries, b, p, nullptr, nullptr, entry_idx, entry_score, entry_weight, lse,
                    static_cast<cudaStream_t>(cuda_stream), nullptr, /*flat=*/true);
}

htam_status htam_query_host(htam_memory *m, const void *queries, int32_t b, const htam_query_params *p,
                            int32_t *group_idx, float *group_score, int32_t *entry_idx, float *entry_score,
                            float *entry_weight, float *lse, void *cuda_stream) {
  htam_status s = check_query_args(m, queries, b, p, group_idx, group_score, entry_idx, entry_score, entry_weight);
  if (s != HTAM_OK) return s;
  if (b == 0) return HTAM_OK;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const int kg = p->k_groups, ke = p->k_entries;
  const size_t qbytes = (size_t)b * m->d * m->elem_bytes;
  const size_t bytes = Carver::round(qbytes) + 2 * Carver::round((size_t)b * kg * 4) +
                       3 * Carver::round((size_t)b * ke * 4) + Carver::round((size_t)b * 4) + 1024;
  if (bytes > m->stage_bytes) {
    if (m->stage) cudaFree(m->stage);
    m->stage = nullptr;
    m->stage_bytes = 0;
    if (cudaMalloc(&m->stage, bytes) != cudaSuccess) {
      cudaGetLastError();
      return HTAM_ENOMEM;
    }
    m->stage_bytes = bytes;
  }
  Carver cv(m->stage);
  void *dq = cv.take<char>(qbytes);
  int32_t *dgi = cv.take<int32_t>((size_t)b * kg);
  float *dgs = cv.take<float>((size_t)b * kg);
  int32_t *dei = cv.take<int32_t>((size_t)b * ke);
  float *des = cv.take<float>((size_t)b * ke);
  float *dew = cv.take<float>((size_t)b * ke);
  float *dl = cv.take<float>((size_t)b);
  HTAM_CK(cudaMemcpyAsync(dq, queries, qbytes, cudaMemcpyHostToDevice, st));
  s = query_impl(m, dq, b, *p, dgi, dgs, dei, des, dew, lse ? dl : nullptr, st);
  if (s != HTAM_OK) return s;
  HTAM_CK(cudaMemcpyAsync(group_idx, dgi, (size_t)b * kg * 4, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaMemcpyAsync(group_score, dgs, (size_t)b * kg * 4, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaMemcpyAsync(entry_idx, dei, (size_t)b * ke * 4, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaMemcpyAsync(entry_score, des, (size_t)b * ke * 4, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaMemcpyAsync(entry_weight, dew, (size_t)b * ke * 4, cudaMemcpyDeviceToHost, st));
  if (lse) HTAM_CK(cudaMemcpyAsync(lse, dl, (size_t)b * 4, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaStreamSynchronize(st));
  return HTAM_OK;
}

htam_status htam_memory_info(const htam_memory *m, int64_t *n, int32_t *d, int32_t *n_groups,
                             int64_t *capacity) {
  if (!m) return HTAM_EINVAL;
  if (n) {
    // The host mirror is a cache of device state: waiting for the last
    // append's copy updates it, not the memory.
    htam_status s = refresh_mirror(const_cast<htam_memory *>(m), true);
    if (s != HTAM_OK) return s;
    *n = m->n;
  }
  if (d) *d = m->d;
  if (n_groups) *n_groups = m->n_groups;
  if (capacity) *capacity = m->capacity;
  return HTAM_OK;
}

htam_status htam_memory_group_counts(const htam_memory *m, int64_t *counts) {
  if (!m || !counts) return HTAM_EINVAL;
  htam_status s = refresh_mirror(const_cast<htam_memory *>(m), true);  // a cache of device state
  if (s != HTAM_OK) return s;
  std::memcpy(counts, m->h_count.data(), sizeof(int64_t) * m->n_groups);
  return HTAM_OK;
}

htam_status htam_memory_group_keys(const htam_memory *m, float *keys, void *cuda_stream) {
  if (!m || !keys) return HTAM_EINVAL;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  HTAM_CK(cudaMemcpyAsync(keys, m->cent, sizeof(float) * (size_t)m->n_groups * m->d, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaStreamSynchronize(st));
  return HTAM_OK;
}

htam_status htam_device_status(htam_memory *m, void *cuda_stream) {
  if (!m) return HTAM_EINVAL;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  unsigned int word = 0;
  HTAM_CK(cudaMemcpyAsync(&word, m->status, sizeof word, cudaMemcpyDeviceToHost, st));
  HTAM_CK(cudaMemsetAsync(m->status, 0, sizeof(unsigned int), st));
  HTAM_CK(cudaStreamSynchronize(st));
  htam_status s = refresh_mirror(m, true);
  if (s != HTAM_OK) return s;
  if (word & 1u) return HTAM_ETIMEOUT;
  if (word & 2u) return HTAM_EINVAL;  // an append was rejected on the device
  return HTAM_OK;
}

htam_status htam_set_tuning(htam_memory *m, htam_tuning key, int32_t value) {
  if (!m) return HTAM_EINVAL;
  switch (key) {
    case HTAM_TUNE_TC_MIN_BUCKET:
      if (value < 1) return HTAM_EINVAL;
      m->tc_min = value;
      return HTAM_OK;
    case HTAM_TUNE_STREAM_ROWS:
      if (value != 0 && value != 1) return HTAM_EINVAL;
      m->stream_rows = value;
      return HTAM_OK;
    case HTAM_TUNE_TC_PAIRS:
      if (value != 0 && value != 1) return HTAM_EINVAL;
      m->tc_pairs = value;
      return HTAM_OK;
    case HTAM_TUNE_PDL:
      if (value != 0 && value != 1) return HTAM_EINVAL;
      m->pdl = value;
      return HTAM_OK;
    case HTAM_TUNE_FINE_OVERLAP:
      if (value != 0 && value != 1) return HTAM_EINVAL;
      m->fine_overlap = value;
      return HTAM_OK;
  }
  return HTAM_EINVAL;
}

htam_status htam_get_tuning(const htam_memory *m, htam_tuning key, int32_t *value) {
  if (!m || !value) return HTAM_EINVAL;
  switch (key) {
    case HTAM_TUNE_TC_MIN_BUCKET:
      *value = m->tc_min;
      return HTAM_OK;
    case HTAM_TUNE_STREAM_ROWS:
      *value = m->stream_rows;
      return HTAM_OK;
    case HTAM_TUNE_TC_PAIRS:
      *value = m->tc_pairs;
      return HTAM_OK;
    case HTAM_TUNE_PDL:
      *value = m->pdl;
      return HTAM_OK;
    case HTAM_TUNE_FINE_OVERLAP:
      *value = m->fine_overlap;
      return HTAM_OK;
  }
  return HTAM_EINVAL;
}

htam_status htam_set_phase_timing(htam_memory *m, int enable) {
  if (!m) return HTAM_EINVAL;
  m->timing = enable != 0;
  return HTAM_OK;
}

htam_status htam_read_phase_timing(htam_memory *m, double *ms, int64_t *launches, int64_t *queries,
                                   void *cuda_stream) {
  if (!m) return HTAM_EINVAL;
  HTAM_CK(cudaStreamSynchronize(static_cast<cudaStream_t>(cuda_stream)));
  double acc[HTAM_N_PHASES] = {};
  for (size_t i = 0; i < m->ev_used / 2; ++i) {
    float t = 0.f;
    HTAM_CK(cudaEventSynchronize(m->ev_pool[2 * i + 1]));
    HTAM_CK(cudaEventElapsedTime(&t, m->ev_pool[2 * i], m->ev_pool[2 * i + 1]));
    acc[m->ev_phase[i]] += t;
  }
  for (int p = 0; p < HTAM_N_PHASES; ++p) {
    if (ms) ms[p] = acc[p];
    if (launches) launches[p] = m->phase_launches[p];
    m->phase_launches[p] = 0;
  }
  if (queries) *queries = m->n_queries;
  m->n_queries = 0;
  m->ev_used = 0;
  m->ev_phase.clear();
  return HTAM_OK;
}

void htam_free_memory(htam_memory *m) { free_impl(m); }

htam_status htam_selftest_wait_timeout(int64_t max_iters, void *cuda_stream) {
  htam_status s = check_device();
  if (s != HTAM_OK) return s;
  if (max_iters < 0) return HTAM_EINVAL;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  unsigned int *buf = nullptr;  // [0] flag nobody sets, [1] status
  HTAM_CK(cudaMalloc(&buf, 2 * sizeof(unsigned int)));
  unsigned int host[2] = {0, 0};
  cudaError_t e = cudaMemsetAsync(buf, 0, 2 * sizeof(unsigned int), st);
  if (e == cudaSuccess) {
    wait_timeout_selftest_kernel<<<1, 32, 0, st>>>(buf, (long long)max_iters, buf + 1);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(host, buf, sizeof host, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(buf);
  if (e != cudaSuccess) {
    set_last_error("htam_selftest_wait_timeout", e);
    return HTAM_ECUDA;
  }
  return host[1] ? HTAM_ETIMEOUT : HTAM_OK;
}

}  // extern "C"
