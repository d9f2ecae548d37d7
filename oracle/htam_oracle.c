/*
 * htam_oracle.c -- float64 brute-force CPU oracle for HTAM's hierarchical
 * transition-attended memory lookup (arxiv 2605.29734).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow definition that the
 * CUDA path is checked against.  Only the tests, the package smoke check and
 * the benchmark's CPU-baseline leg may load it; the product path never does.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * What it computes (one query q, memory of n entries k_e with group ids):
 *   Memory (Eq. 6, §4.1): global nodes V_G = groups, local nodes V_GL =
 *     entries, each entry tagged with its parent group par(e) (Eq. 12).
 *   Group key: c_g = (1/n_g) * sum_{e: par(e)=g} k_e   (mean of its entries;
 *     the paper leaves the embedding of a global node open, the workload
 *     definition fixes it as the mean).
 *   Stage 1 (Eq. 9 with the linear scorer of App. B.6, phi = w^T z; in
 *     embedding space the linear scorer is the dot product):
 *       s1[g] = q . c_g for every non-empty g; S = the k_g best groups,
 *       ordered by score descending, ties to the lower group id.  Empty groups
 *       (n_g = 0) are never candidates (App. B.7: a direction with no valid
 *       local node gives no candidate).
 *   Stage 2 (Eq. 12 restriction, Eq. 13 pick, Eq. 11 policy):
 *       C = { e : par(e) in S }  (candidate restriction L(g_t)),
 *       s2[e] = q . k_e for e in C,
 *       lse = log sum_{e in C} exp(s2[e]/tau),
 *       w[e] = eps/|C| + (1-eps) * exp(s2[e]/tau - lse)   (the eps-uniform /
 *         tau-softmax mixture of Eq. 11, normalised over the whole candidate
 *         set C),
 *       output: the k_e best e of C by s2 descending, ties to the lower entry
 *       id, with s2 and w; slots beyond |C| are padded with id -1, score
 *       -inf, weight 0.
 *
 * Everything is double precision, sequential sums in index order, brute force
 * over the caller's arrays in their original (unsorted) order.  Inputs are
 * float32 (dtype 0) or bfloat16 bit patterns (dtype 1, uint16), converted
 * exactly to double.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_F32 0
#define ORACLE_BF16 1

/* Exact conversion of element idx of an fp32 or bf16 array to double. */
static double load_elem(const void *base, int dtype, int64_t idx) {
  if (dtype == ORACLE_F32) {
    return (double)((const float *)base)[idx];
  }
  uint16_t bits = ((const uint16_t *)base)[idx];
  uint32_t wide = ((uint32_t)bits) << 16;
  float f;
  memcpy(&f, &wide, sizeof f);
  return (double)f;
}

/* ---------------------------------------------------------------- centroids
 * Adds every entry of the chunk into sums[gid][:] and counts[gid].  Callers
 * zero sums/counts first and may feed the entries in several chunks.  Threads
 * split the coordinates, so each sums[g][j] is still added in entry order.
 * Returns 0, or -1 when a group id is outside [0, n_groups). */
typedef struct {
  const void *entries;
  int dtype;
  const int32_t *gid;
  int64_t n;
  int32_t d, j0, j1;
  double *sums;
} centroid_job;

static void *centroid_worker(void *arg) {
  centroid_job *job = (centroid_job *)arg;
  for (int64_t e = 0; e < job->n; ++e) {
    double *row = job->sums + (int64_t)job->gid[e] * job->d;
    for (int32_t j = job->j0; j < job->j1; ++j) {
      row[j] += load_elem(job->entries, job->dtype, e * (int64_t)job->d + j);
    }
  }
  return NULL;
}

int htam_oracle_centroid_accumulate(const void *entries, int dtype,
                                    const int32_t *gid, int64_t n, int32_t d,
                                    int32_t n_groups, double *sums,
                                    int64_t *counts, int nthreads) {
  for (int64_t e = 0; e < n; ++e) {
    if (gid[e] < 0 || gid[e] >= n_groups) return -1;
  }
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (nthreads > d) nthreads = d;
  centroid_job jobs[256];
  pthread_t threads[256];
  int started[256];
  for (int t = 0; t < nthreads; ++t) {
    centroid_job j = {entries, dtype, gid, n, d, (int32_t)((int64_t)d * t / nthreads),
                      (int32_t)((int64_t)d * (t + 1) / nthreads), sums};
    jobs[t] = j;
    started[t] = 0;
  }
  for (int t = 1; t < nthreads; ++t) {
    started[t] = pthread_create(&threads[t], NULL, centroid_worker, &jobs[t]) == 0;
    if (!started[t]) centroid_worker(&jobs[t]);
  }
  centroid_worker(&jobs[0]);
  for (int t = 1; t < nthreads; ++t) {
    if (started[t]) pthread_join(threads[t], NULL);
  }
  for (int64_t e = 0; e < n; ++e) counts[gid[e]] += 1;
  return 0;
}

/* c_g = sums_g / n_g; groups with n_g = 0 are left as NaN (never used). */
void htam_oracle_centroid_finalize(const double *sums, const int64_t *counts,
                                   int32_t d, int32_t n_groups,
                                   double *centroid) {
  for (int32_t g = 0; g < n_groups; ++g) {
    for (int32_t j = 0; j < d; ++j) {
      centroid[(int64_t)g * d + j] =
          counts[g] > 0 ? sums[(int64_t)g * d + j] / (double)counts[g] : NAN;
    }
  }
}

/* ------------------------------------------------------------- ordering */
typedef struct {
  double score;
  int64_t id;
} scored_t;

/* Score descending, then id ascending. */
static int by_score_then_id(const void *pa, const void *pb) {
  const scored_t *a = (const scored_t *)pa;
  const scored_t *b = (const scored_t *)pb;
  if (a->score > b->score) return -1;
  if (a->score < b->score) return 1;
  if (a->id < b->id) return -1;
  if (a->id > b->id) return 1;
  return 0;
}

/* ------------------------------------------------------------- stage 1 */
typedef struct {
  const void *queries;
  int q_dtype;
  int32_t n_queries, d;
  const double *centroid;
  const int64_t *counts;
  int32_t n_groups, k_groups;
  int32_t *group_idx;
  double *group_score;
  int tid, nthreads;
  int status;
} stage1_job;

static void *stage1_worker(void *arg) {
  stage1_job *job = (stage1_job *)arg;
  scored_t *cand = (scored_t *)malloc(sizeof(scored_t) * (size_t)job->n_groups);
  if (!cand) {
    job->status = -2;
    return NULL;
  }
  for (int32_t b = job->tid; b < job->n_queries; b += job->nthreads) {
    int32_t n_cand = 0;
    for (int32_t g = 0; g < job->n_groups; ++g) {
      if (job->counts[g] == 0) continue;
      double s = 0.0;
      for (int32_t j = 0; j < job->d; ++j) {
        s += load_elem(job->queries, job->q_dtype, (int64_t)b * job->d + j) *
             job->centroid[(int64_t)g * job->d + j];
      }
      cand[n_cand].score = s;
      cand[n_cand].id = g;
      ++n_cand;
    }
    qsort(cand, (size_t)n_cand, sizeof(scored_t), by_score_then_id);
    for (int32_t j = 0; j < job->k_groups; ++j) {
      int64_t o = (int64_t)b * job->k_groups + j;
      if (j < n_cand) {
        job->group_idx[o] = (int32_t)cand[j].id;
        job->group_score[o] = cand[j].score;
      } else {
        job->group_idx[o] = -1;
        job->group_score[o] = -INFINITY;
      }
    }
  }
  free(cand);
  return NULL;
}

/* ------------------------------------------------------------- stage 2 */
typedef struct {
  const void *entries;
  int e_dtype;
  const int32_t *gid;
  int64_t n;
  int32_t d, n_groups;
  const void *queries;
  int q_dtype;
  int32_t n_queries;
  const int32_t *groups; /* [n_queries, k_groups], -1 = unused slot */
  int32_t k_groups, k_entries;
  double tau, eps;
  int32_t *entry_idx;
  double *entry_score, *entry_weight, *lse;
  int64_t *n_cand_out;
  int tid, nthreads;
  int status;
} stage2_job;

static void *stage2_worker(void *arg) {
  stage2_job *job = (stage2_job *)arg;
  unsigned char *selected = (unsigned char *)malloc((size_t)job->n_groups);
  scored_t *cand = (scored_t *)malloc(sizeof(scored_t) * (size_t)(job->n > 0 ? job->n : 1));
  if (!selected || !cand) {
    free(selected);
    free(cand);
    job->status = -2;
    return NULL;
  }
  for (int32_t b = job->tid; b < job->n_queries; b += job->nthreads) {
    memset(selected, 0, (size_t)job->n_groups);
    for (int32_t j = 0; j < job->k_groups; ++j) {
      int32_t g = job->groups[(int64_t)b * job->k_groups + j];
      if (g >= 0 && g < job->n_groups) selected[g] = 1;
    }
    /* Candidate restriction: entries whose parent group was selected. */
    int64_t n_cand = 0;
    for (int64_t e = 0; e < job->n; ++e) {
      if (!selected[job->gid[e]]) continue;
      double s = 0.0;
      for (int32_t j = 0; j < job->d; ++j) {
        s += load_elem(job->queries, job->q_dtype, (int64_t)b * job->d + j) *
             load_elem(job->entries, job->e_dtype, e * (int64_t)job->d + j);
      }
      cand[n_cand].score = s;
      cand[n_cand].id = e;
      ++n_cand;
    }
    /* Softmax over the whole candidate set, max-shifted. */
    double lse_b = -INFINITY;
    if (n_cand > 0) {
      double m = -INFINITY;
      for (int64_t i = 0; i < n_cand; ++i) {
        double z = cand[i].score / job->tau;
        if (z > m) m = z;
      }
      double sum = 0.0;
      for (int64_t i = 0; i < n_cand; ++i) {
        sum += exp(cand[i].score / job->tau - m);
      }
      lse_b = m + log(sum);
    }
    qsort(cand, (size_t)n_cand, sizeof(scored_t), by_score_then_id);
    for (int32_t j = 0; j < job->k_entries; ++j) {
      int64_t o = (int64_t)b * job->k_entries + j;
      if (j < n_cand) {
        job->entry_idx[o] = (int32_t)cand[j].id;
        job->entry_score[o] = cand[j].score;
        job->entry_weight[o] =
            job->eps / (double)n_cand +
            (1.0 - job->eps) * exp(cand[j].score / job->tau - lse_b);
      } else {
        job->entry_idx[o] = -1;
        job->entry_score[o] = -INFINITY;
        job->entry_weight[o] = 0.0;
      }
    }
    job->lse[b] = lse_b;
    job->n_cand_out[b] = n_cand;
  }
  free(selected);
  free(cand);
  return NULL;
}

static int clamp_threads(int nthreads, int32_t n_queries) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (n_queries > 0 && nthreads > n_queries) nthreads = n_queries;
  return nthreads;
}

/* Stage 1 for n_queries queries.  centroid [n_groups, d], counts [n_groups].
 * Outputs group_idx [n_queries, k_groups] and group_score (same shape).
 * Returns 0, -1 on bad arguments, -2 on allocation failure. */
int htam_oracle_stage1(const void *queries, int q_dtype, int32_t n_queries,
                       int32_t d, const double *centroid,
                       const int64_t *counts, int32_t n_groups,
                       int32_t k_groups, int32_t *group_idx,
                       double *group_score, int nthreads) {
  if (n_queries < 0 || d <= 0 || n_groups <= 0 || k_groups <= 0) return -1;
  nthreads = clamp_threads(nthreads, n_queries);
  stage1_job jobs[256];
  pthread_t threads[256];
  for (int t = 0; t < nthreads; ++t) {
    stage1_job j = {queries, q_dtype, n_queries, d, centroid, counts,
                    n_groups, k_groups, group_idx, group_score, t, nthreads, 0};
    jobs[t] = j;
  }
  for (int t = 1; t < nthreads; ++t) {
    if (pthread_create(&threads[t], NULL, stage1_worker, &jobs[t]) != 0) {
      jobs[t].status = -3;
    }
  }
  stage1_worker(&jobs[0]);
  int status = jobs[0].status;
  for (int t = 1; t < nthreads; ++t) {
    if (jobs[t].status != -3) pthread_join(threads[t], NULL);
    if (jobs[t].status != 0) status = jobs[t].status;
  }
  return status;
}

/* Stage 2 for n_queries queries given each query's selected groups
 * (groups [n_queries, k_groups], -1 for unused slots).  Outputs entry_idx,
 * entry_score, entry_weight [n_queries, k_entries], lse [n_queries] and the
 * candidate-set size n_cand [n_queries].  Returns 0, -1 on bad arguments
 * (including a group id outside [0, n_groups)), -2 on allocation failure. */
int htam_oracle_stage2(const void *entries, int e_dtype, const int32_t *gid,
                       int64_t n, int32_t d, int32_t n_groups,
                       const void *queries, int q_dtype, int32_t n_queries,
                       const int32_t *groups, int32_t k_groups,
                       int32_t k_entries, double tau, double eps,
                       int32_t *entry_idx, double *entry_score,
                       double *entry_weight, double *lse, int64_t *n_cand,
                       int nthreads) {
  if (n < 0 || d <= 0 || n_groups <= 0 || n_queries < 0 || k_groups <= 0 ||
      k_entries <= 0 || !(tau > 0.0) || !(eps >= 0.0 && eps <= 1.0)) {
    return -1;
  }
  for (int64_t e = 0; e < n; ++e) {
    if (gid[e] < 0 || gid[e] >= n_groups) return -1;
  }
  nthreads = clamp_threads(nthreads, n_queries);
  stage2_job jobs[256];
  pthread_t threads[256];
  for (int t = 0; t < nthreads; ++t) {
    stage2_job j = {entries, e_dtype, gid, n, d, n_groups, queries, q_dtype,
                    n_queries, groups, k_groups, k_entries, tau, eps,
                    entry_idx, entry_score, entry_weight, lse, n_cand, t,
                    nthreads, 0};
    jobs[t] = j;
  }
  for (int t = 1; t < nthreads; ++t) {
    if (pthread_create(&threads[t], NULL, stage2_worker, &jobs[t]) != 0) {
      jobs[t].status = -3;
    }
  }
  stage2_worker(&jobs[0]);
  int status = jobs[0].status;
  for (int t = 1; t < nthreads; ++t) {
    if (jobs[t].status != -3) pthread_join(threads[t], NULL);
    if (jobs[t].status != 0) status = jobs[t].status;
  }
  return status;
}

/* ------------------------------------------------------- prefix query (N1)
 * A prefix-attended query (Eq. 9 summed over the global prefix of
 * Eq. 8 with the position-aware weights of Eq. 10): for a prefix of P state
 * embeddings q_1..q_P (q_P the most recent),
 *   score(g) = sum_{i=1..P} alpha_i * (q_i . c_g),
 *   alpha_i  = exp(-lambda * (P - i)).
 * The scorer is linear in the query, so score(g) = qbar . c_g with
 *   qbar = sum_{i=1..P} alpha_i * q_i,
 * and the rest of the lookup runs on qbar.  This writes qbar in double:
 * prefix [n_queries, p_len, d] (dtype 0 fp32, 1 bf16 bits), out
 * [n_queries, d]; the sum runs over i = 1..P in order.  Returns 0, or -1 on a
 * bad argument. */
int htam_oracle_prefix_reduce(const void *prefix, int dtype, int32_t n_queries, int32_t p_len, int32_t d,
                              double lambda, double *out) {
  if (n_queries < 0 || p_len < 1 || d < 1 || !(lambda >= 0.0)) return -1;
  for (int32_t b = 0; b < n_queries; ++b) {
    double *o = out + (int64_t)b * d;
    for (int32_t j = 0; j < d; ++j) o[j] = 0.0;
    for (int32_t i = 1; i <= p_len; ++i) {
      const double alpha = exp(-lambda * (double)(p_len - i));
      const int64_t row = ((int64_t)b * p_len + (i - 1)) * d;
      for (int32_t j = 0; j < d; ++j) o[j] += alpha * load_elem(prefix, dtype, row + j);
    }
  }
  return 0;
}

/* ------------------------------------------------ edge-table routing (N2)
 * The global router of Eq. 9 with the transition utility of App. B.6: the
 * utility of moving from direction g_i to direction g is a fixed linear
 * reward over the edge's feature vector, phi(g_i, g) = w . z(g_i, g).  The
 * features come from a table Z [G, G, F] of float32 (row = from, column =
 * to).  For a prefix p_1..p_P of earlier group ids per query (-1 = no
 * element, contributes nothing) and the weights alpha_i = exp(-lambda (P - i))
 * of Eq. 10,
 *   score[b][g] = sum_{i = 1..P, p_i >= 0} alpha_i * sum_{f} w_f Z[p_i][g][f],
 * summed in index order in double.  Returns 0, or -1 on a bad argument. */
int htam_oracle_edge_scores(const float *Z, int32_t G, int32_t F, const double *w, const int32_t *prefix,
                            int32_t n_queries, int32_t p_len, double lambda, double *out) {
  if (G < 1 || F < 1 || n_queries < 0 || p_len < 1 || !(lambda >= 0.0)) return -1;
  for (int32_t b = 0; b < n_queries; ++b) {
    double *o = out + (int64_t)b * G;
    for (int32_t g = 0; g < G; ++g) o[g] = 0.0;
    for (int32_t i = 1; i <= p_len; ++i) {
      const int32_t from = prefix[(int64_t)b * p_len + (i - 1)];
      if (from < 0) continue;
      if (from >= G) return -1;
      const double alpha = exp(-lambda * (double)(p_len - i));
      for (int32_t g = 0; g < G; ++g) {
        const float *z = Z + ((int64_t)from * G + g) * F;
        double phi = 0.0;
        for (int32_t f = 0; f < F; ++f) phi += w[f] * (double)z[f];
        o[g] += alpha * phi;
      }
    }
  }
  return 0;
}

/* The k best groups of given per-group scores, ranked as stage 1 ranks them:
 * score descending, ties to the lower group id, empty groups (counts 0)
 * never candidates, -1 / -inf padding.  Returns 0, or -2 on allocation
 * failure. */
int htam_oracle_select(const double *scores, const int64_t *counts, int32_t n_queries, int32_t G, int32_t k,
                       int32_t *group_idx, double *group_score) {
  scored_t *cand = (scored_t *)malloc(sizeof(scored_t) * (size_t)G);
  if (!cand) return -2;
  for (int32_t b = 0; b < n_queries; ++b) {
    int32_t n_cand = 0;
    for (int32_t g = 0; g < G; ++g) {
      if (counts[g] == 0) continue;
      cand[n_cand].score = scores[(int64_t)b * G + g];
      cand[n_cand].id = g;
      ++n_cand;
    }
    qsort(cand, (size_t)n_cand, sizeof(scored_t), by_score_then_id);
    for (int32_t j = 0; j < k; ++j) {
      const int64_t o = (int64_t)b * k + j;
      group_idx[o] = j < n_cand ? (int32_t)cand[j].id : -1;
      group_score[o] = j < n_cand ? cand[j].score : -INFINITY;
    }
  }
  free(cand);
  return 0;
}

/* ------------------------------------------------------------------------
 * Sampling from the global-direction policy (Eq. 11; Algorithm 1, step 2
 * draws g_t from it).
 *
 * Generator: Philox4x32-10, the counter-based generator of Salmon, Moraes,
 * Dror and Shaw ("Parallel random numbers: as easy as 1, 2, 3", SC 2011).
 * A 128-bit counter (four 32-bit words) and a 64-bit key (two words) map to
 * four 32-bit outputs through ten rounds.  A round multiplies counter words 0
 * and 2 by two fixed odd constants, giving 64-bit products; the new words are
 * (high half of product 2) xor word 1 xor key 0, (low half of product 2),
 * (high half of product 0) xor word 3 xor key 1, (low half of product 0).
 * Between rounds both key words advance by fixed Weyl increments (the golden
 * ratio and sqrt(3) - 1, scaled to 32 bits). */
static const uint32_t kPhiloxMul0 = 0xD2511F53u, kPhiloxMul1 = 0xCD9E8D57u;
static const uint32_t kPhiloxWeyl0 = 0x9E3779B9u, kPhiloxWeyl1 = 0xBB67AE85u;

void htam_oracle_philox4x32_10(const uint32_t *ctr, const uint32_t *key, uint32_t *out) {
  uint32_t c[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += kPhiloxWeyl0;
      k1 += kPhiloxWeyl1;
    }
    const uint64_t p0 = (uint64_t)kPhiloxMul0 * c[0];
    const uint64_t p1 = (uint64_t)kPhiloxMul1 * c[2];
    const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c[1] ^ k0;
    const uint32_t n1 = (uint32_t)p1;
    const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c[3] ^ k1;
    const uint32_t n3 = (uint32_t)p0;
    c[0] = n0;
    c[1] = n1;
    c[2] = n2;
    c[3] = n3;
  }
  out[0] = c[0];
  out[1] = c[1];
  out[2] = c[2];
  out[3] = c[3];
}

/* The uniform of query b and group g: word (g mod 4) of Philox4x32-10 at
 * counter (g / 4, b, low and high words of `offset`) under key (low and high
 * words of `seed`); its top 23 bits plus one half, times 2^-23, so that
 * u lies in (0, 1) and is exact in float32. */
double htam_oracle_policy_uniform(uint64_t seed, uint64_t offset, int32_t b, int32_t g) {
  const uint32_t ctr[4] = {(uint32_t)g >> 2, (uint32_t)b, (uint32_t)offset, (uint32_t)(offset >> 32)};
  const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t out[4];
  htam_oracle_philox4x32_10(ctr, key, out);
  return ((double)(out[g & 3] >> 9) + 0.5) * (1.0 / 8388608.0);
}

/* The policy of Eq. 11 over the candidate directions G_t = the non-empty
 * groups (n of them), and the keys that draw from it.
 *   mu[b][g] = eps / n + (1 - eps) * exp(s[b][g] / tau - lse_b),
 *   lse_b = log sum_{g in G_t} exp(s[b][g] / tau)
 * (0 for empty groups).  keys[b][g] = log mu[b][g] - log(-log u(b, g)) (log mu
 * taken as s/tau - lse when eps = 0; -inf for empty groups).  The k groups
 * with the largest keys (ties to the lower id) are k draws without
 * replacement from mu, in draw order: the Gumbel-top-k construction (Kool, van
 * Hoof and Welling, ICML 2019; k = 1 is the Gumbel-max draw of g_t ~ mu).
 * Row b uses the uniforms of query query_ids[b] (of query b when query_ids
 * is NULL), so that a sample of a batch's rows draws what the whole batch
 * draws.  Returns 0, or -1 on a bad argument. */
int htam_oracle_policy_keys(const double *scores, const int64_t *counts, int32_t n_queries, int32_t G, double tau,
                            double eps, uint64_t seed, uint64_t offset, const int32_t *query_ids, double *keys,
                            double *mu) {
  if (G < 1 || n_queries < 0 || !(tau > 0.0) || !(eps >= 0.0 && eps <= 1.0)) return -1;
  int64_t n = 0;
  for (int32_t g = 0; g < G; ++g) n += counts[g] > 0;
  for (int32_t b = 0; b < n_queries; ++b) {
    const double *s = scores + (int64_t)b * G;
    double m = -INFINITY;
    for (int32_t g = 0; g < G; ++g) {
      if (counts[g] > 0 && s[g] / tau > m) m = s[g] / tau;
    }
    double sum = 0.0;
    for (int32_t g = 0; g < G; ++g) {
      if (counts[g] > 0) sum += exp(s[g] / tau - m);
    }
    const double lse = m + log(sum);
    for (int32_t g = 0; g < G; ++g) {
      const int64_t o = (int64_t)b * G + g;
      if (counts[g] == 0) {
        mu[o] = 0.0;
        keys[o] = -INFINITY;
        continue;
      }
      mu[o] = eps / (double)n + (1.0 - eps) * exp(s[g] / tau - lse);
      const double log_mu = eps == 0.0 ? s[g] / tau - lse : log(mu[o]);
      const double u = htam_oracle_policy_uniform(seed, offset, query_ids ? query_ids[b] : b, g);
      keys[o] = log_mu - log(-log(u));
    }
  }
  return 0;
}
