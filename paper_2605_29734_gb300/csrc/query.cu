// query.cu -- the two-level lookup (read side of one evolution step, §4.3).
//
//   1. coarse scores s1[b][g] = q_b . c_g against every group key (Eq. 9
//      with the linear scorer of App. B.6) and the k_groups best groups;
//   2. bucketing: invert query -> selected groups into group -> queries so
//      that each selected group's pages are streamed once per bucket chunk;
//   3. fine scores over the entries of the selected groups only (the Eq. 12
//      restriction), with the per-query online softmax statistics (Eq. 11)
//      and a running top-k_entries (Eq. 13 as a top-k) fused in;
//   4. merge of the per-unit partial results per query: log-sum-exp combine,
//      final top-k, weights eps/|C| + (1-eps) exp(s/tau - lse).
// Nothing is read back to the host; every size that depends on the data
// lives on the device and the kernels loop over it.

#include <algorithm>
#include <cstring>
#include <vector>

#include "common.cuh"
#include "coarse_tc.h"
#include "fine_stream.h"
#include "fine_tc.h"
#include "internal.h"

namespace htam {

namespace {

// ------------------------------------------------------------------ stage 1

// s1[b][g] = q_b . cent_g in fp32; -inf for empty groups.  64x64 tile per
// block, 16x16 threads with 4x4 outputs each, k-slices of 32 staged in
// shared memory.
template <typename T>
__global__ void __launch_bounds__(256) coarse_scores_simt_kernel(
    const T *__restrict__ Q, int B, int d, const float *__restrict__ cent,
    const int32_t *__restrict__ count, int G, float *__restrict__ s1, const int32_t *__restrict__ gate = nullptr) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  if (gate && *gate == 0) return;  // gated launch with nothing to score
  __shared__ float qs[32][68];
  __shared__ float cs[32][68];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int b0 = blockIdx.y * 64, g0 = blockIdx.x * 64;
  float acc[4][4] = {};
  const int lr = tid >> 2, lc = (tid & 3) * 8;  // loader: row, 8 columns
  for (int k0 = 0; k0 < d; k0 += 32) {
    {
      int b = b0 + lr, k = k0 + lc;
      float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      if (b < B && k < d) {
        const T *p = Q + (int64_t)b * d + k;
        if constexpr (sizeof(T) == 2) {
          uint4 w = *reinterpret_cast<const uint4 *>(p);
          v[0] = bf16lo(w.x); v[1] = bf16hi(w.x); v[2] = bf16lo(w.y); v[3] = bf16hi(w.y);
          v[4] = bf16lo(w.z); v[5] = bf16hi(w.z); v[6] = bf16lo(w.w); v[7] = bf16hi(w.w);
        } else {
          float4 a = *reinterpret_cast<const float4 *>(p);
          float4 c = *reinterpret_cast<const float4 *>(p + 4);
          v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = c.x; v[5] = c.y; v[6] = c.z; v[7] = c.w;
        }
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) qs[lc + i][lr] = v[i];
    }
    {
      int g = g0 + lr, k = k0 + lc;
      float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      if (g < G && k < d) {
        const float *p = cent + (int64_t)g * d + k;
        float4 a = *reinterpret_cast<const float4 *>(p);
        float4 c = *reinterpret_cast<const float4 *>(p + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = c.x; v[5] = c.y; v[6] = c.z; v[7] = c.w;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) cs[lc + i][lr] = v[i];
    }
    __syncthreads();
#pragma unroll 8
    for (int k = 0; k < 32; ++k) {
      float4 a = *reinterpret_cast<const float4 *>(&qs[k][ty * 4]);
      float4 c = *reinterpret_cast<const float4 *>(&cs[k][tx * 4]);
      float av[4] = {a.x, a.y, a.z, a.w}, cv[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], cv[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int b = b0 + ty * 4 + i;
    if (b >= B) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int g = g0 + tx * 4 + j;
      if (g < G) s1[(int64_t)b * G + g] = count[g] > 0 ? acc[i][j] : -INFINITY;
    }
  }
}

// A team of WPQ warps per query (8 warps per block): top-k_groups of
// sum_z s1[z][b][:] (score desc, lower g on ties), empty groups excluded;
// -1 / -inf padding.  Each warp keeps the top-k of its share of the groups,
// loading kSelBatch chunks of 32 scores per lane before comparing any; the
// team's first warp then merges the team's lists.  Few queries take teams of
// eight warps so that the grid fills the GPU; many take one warp each.
constexpr int kSelWarps = 8;
constexpr int kSelBatch = 8;
constexpr int kSelSortMin = 4;  // more candidates than this in a chunk: sort and merge

template <int WPQ, int NW = (WPQ > kSelWarps ? WPQ : kSelWarps)>
__global__ void __launch_bounds__(NW * 32, 1) group_topk_kernel(const float *__restrict__ s1, int planes,
                                                             int B, int G,
                                                             const int32_t *__restrict__ count, int kg,
                                                             int32_t *__restrict__ gidx,
                                                             float *__restrict__ gscore,
                                                             const int32_t *__restrict__ gate = nullptr) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  if (gate && *gate == 0) return;  // gated launch with nothing to select
  __shared__ float ls[NW][64];
  __shared__ int li[NW][64];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * (NW / WPQ) + warp / WPQ;
  const int sw = warp % WPQ;  // this warp's place in the team
  const bool live = b < B;    // uniform per warp
  const int64_t plane = (int64_t)B * G;
  const float *row = s1 + (int64_t)(live ? b : 0) * G;
  constexpr int kStep = WPQ * 32;
  WarpList L;
  L.init();
  float ts = -INFINITY;
  int ti = INT_MAX;
  for (int base = sw * 32; live && base < G; base += kStep * kSelBatch) {
    float sv[kSelBatch];
    int cv[kSelBatch];
#pragma unroll
    for (int u = 0; u < kSelBatch; ++u) {
      const int g = base + u * kStep + lane;
      cv[u] = g < G ? count[g] : 0;
      sv[u] = g < G ? row[g] : -INFINITY;
    }
    for (int z = 1; z < planes; ++z) {
#pragma unroll
      for (int u = 0; u < kSelBatch; ++u) {
        const int g = base + u * kStep + lane;
        if (g < G) sv[u] += row[z * plane + g];
      }
    }
#pragma unroll
    for (int u = 0; u < kSelBatch; ++u) {
      const int g0 = base + u * kStep;
      const bool valid = cv[u] > 0;
      const float sc = valid ? sv[u] : -INFINITY;
      const bool pass = valid && better(sc, g0 + lane, ts, ti);
      unsigned mask = __ballot_sync(kFullMask, pass);
      if (kg <= 32 && __popc(mask) > kSelSortMin) {
        // Many candidates (the list is still filling): sort the chunk across
        // the warp and merge it whole.
        float cs = pass ? sc : -INFINITY;
        int ci = pass ? g0 + lane : INT_MAX;
        warp_sort32(cs, ci);
        L.merge32(cs, ci);
        L.kth(kg, ts, ti);
        continue;
      }
      while (mask) {
        const int src = __ffs(mask) - 1;
        mask &= mask - 1;
        const float cs = __shfl_sync(kFullMask, sc, src);
        L.insert(kg, cs, g0 + src);
        L.kth(kg, ts, ti);
      }
    }
  }
  if constexpr (WPQ > 1) {
    ls[warp][lane] = L.s0;
    li[warp][lane] = L.i0;
    ls[warp][lane + 32] = L.s1;
    li[warp][lane + 32] = L.i1;
    __syncthreads();
    if (sw != 0 || !live) return;
    L.init();
    ts = -INFINITY;
    ti = INT_MAX;
    for (int w = warp; w < warp + WPQ; ++w) {
      if (kg <= 32) {
        // The team's lists are sorted: merge each whole unless its best
        // cannot enter the top-kg.
        const float cs = ls[w][lane];
        const int ci = li[w][lane];
        const float bs = __shfl_sync(kFullMask, cs, 0);
        const int bi = __shfl_sync(kFullMask, ci, 0);
        if (bi != INT_MAX && better(bs, bi, ts, ti)) {
          L.merge32(cs, ci);
          L.kth(kg, ts, ti);
        }
        continue;
      }
      for (int h = 0; h < 2 && h * 32 < kg; ++h) {
        const float cs = ls[w][h * 32 + lane];
        const int ci = li[w][h * 32 + lane];
        unsigned mask = __ballot_sync(kFullMask, h * 32 + lane < kg && ci != INT_MAX && better(cs, ci, ts, ti));
        while (mask) {
          const int src = __ffs(mask) - 1;
          mask &= mask - 1;
          L.insert(kg, __shfl_sync(kFullMask, cs, src), __shfl_sync(kFullMask, ci, src));
          L.kth(kg, ts, ti);
        }
      }
    }
  }
  if (!live) return;
  if (lane < kg) {
    gidx[(int64_t)b * kg + lane] = L.i0 == INT_MAX ? -1 : L.i0;
    gscore[(int64_t)b * kg + lane] = L.i0 == INT_MAX ? -INFINITY : L.s0;
  }
  if (lane + 32 < kg) {
    gidx[(int64_t)b * kg + lane + 32] = L.i1 == INT_MAX ? -1 : L.i1;
    gscore[(int64_t)b * kg + lane + 32] = L.i1 == INT_MAX ? -INFINITY : L.s1;
  }
}

// Warps per query for B queries: eight while B * 8 warps stay under about
// two full waves of the GPU (16 warps per SM), else one.
static int warps_per_query(int B, int sm_count) { return (int64_t)B * 8 <= 2LL * 16 * sm_count ? 8 : 1; }
// Group selection: teams of 32 warps (one 1,024-thread block per query) when
// the batch has no more queries than there are SMs.
// Between those, teams of two warps while B * 2 warps stay under two waves
// (the 1,024-query streaming batches: select 0.018 -> 0.015 ms; one warp
// stays faster at 4,096 queries).
static int select_warps_per_query(int B, int sm_count) {
  if ((int64_t)B <= sm_count) return 32;
  const int w = warps_per_query(B, sm_count);
  return w == 1 && (int64_t)B * 2 <= 2LL * 16 * sm_count ? 2 : w;
}

// Stage-1 scores from a transition-edge table (the router of Eq. 9 with the
// linear utility of App. B.6 and the weights of Eq. 10): one thread per
// (query, group), s1[b][g] = sum_i alpha_i sum_f w_f Z[p_i][g][f] over the
// prefix ids p_i >= 0, in index order with fp32 FMAs.  The threads of a warp
// read neighbouring groups of the same table row, so the loads coalesce.
struct EdgeKernelArgs {
  const float *Z;
  const int32_t *prefix;
  int F, P;
  float w[HTAM_MAX_EDGE_FEATURES];
  float alpha[HTAM_MAX_PREFIX];
};

// phi(from, to) = w . Z[from][to][:], in the same FMA order as below.
__device__ __forceinline__ float edge_phi(const EdgeKernelArgs &a, const float *z) {
  float phi = 0.f;
  if ((a.F & 3) == 0) {
    for (int f = 0; f < a.F; f += 4) {
      const float4 v = *reinterpret_cast<const float4 *>(z + f);
      phi = fmaf(a.w[f], v.x, phi);
      phi = fmaf(a.w[f + 1], v.y, phi);
      phi = fmaf(a.w[f + 2], v.z, phi);
      phi = fmaf(a.w[f + 3], v.w, phi);
    }
  } else {
    for (int f = 0; f < a.F; ++f) phi = fmaf(a.w[f], z[f], phi);
  }
  return phi;
}

// When a batch references more prefix rows than the table has, the utility
// of every edge is formed once (U[from][to] = phi) and the scores gather
// from U: the same products and sums in the same order, so the same results.
__global__ void __launch_bounds__(256) edge_phi_kernel(EdgeKernelArgs a, int G, float *__restrict__ U) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t >= (int64_t)G * G) return;
  U[t] = edge_phi(a, a.Z + t * a.F);
}

__global__ void __launch_bounds__(256) edge_gather_kernel(EdgeKernelArgs a, const float *__restrict__ U, int B, int G,
                                                          float *__restrict__ s1) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * G) return;
  const int64_t b = t / G;
  const int g = (int)(t % G);
  float acc = 0.f;
  for (int i = 0; i < a.P; ++i) {
    const int from = a.prefix[b * a.P + i];
    if (from >= 0) acc = fmaf(a.alpha[i], U[(int64_t)from * G + g], acc);
  }
  s1[t] = acc;
}

__global__ void __launch_bounds__(256) edge_scores_kernel(EdgeKernelArgs a, int B, int G, float *__restrict__ s1) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * G) return;
  const int64_t b = t / G;
  const int g = (int)(t % G);
  float acc = 0.f;
  for (int i = 0; i < a.P; ++i) {
    const int from = a.prefix[b * a.P + i];
    if (from < 0) continue;
    acc = fmaf(a.alpha[i], edge_phi(a, a.Z + ((int64_t)from * G + g) * a.F), acc);
  }
  s1[t] = acc;
}

// ------------------------------------------------------- policy draws (Eq. 11)

// Philox4x32-10 (Salmon, Moraes, Dror and Shaw, SC 2011): ten rounds of two
// 32x32 -> 64-bit products of counter words 0 and 2, mixed with the other
// words and the key; the key advances by two Weyl increments between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k.x += 0x9E3779B9u;
      k.y += 0xBB67AE85u;
    }
    const uint32_t p0_hi = __umulhi(0xD2511F53u, c.x), p0_lo = 0xD2511F53u * c.x;
    const uint32_t p1_hi = __umulhi(0xCD9E8D57u, c.z), p1_lo = 0xCD9E8D57u * c.z;
    c = make_uint4(p1_hi ^ c.y ^ k.x, p1_lo, p0_hi ^ c.w ^ k.y, p0_lo);
  }
  return c;
}

struct PolicyArgs {
  const float *s1;  // [planes, B, G] scores, summed over the planes in order
  int planes, B, G;
  const int32_t *count;
  int n_nonempty;   // |G_t|
  float inv_tau, eps;
  uint2 key;        // seed words
  uint32_t off_lo, off_hi;
  float *keys;      // [B, G] out
};

__device__ __forceinline__ float block_reduce(float v, bool is_max, float *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float w = __shfl_xor_sync(kFullMask, v, o);
    v = is_max ? fmaxf(v, w) : v + w;
  }
  __syncthreads();  // the previous reduction's readers are done with red
  if (lane == 0) red[warp] = v;
  __syncthreads();
  v = red[0];
  for (int w = 1; w < (int)(blockDim.x >> 5); ++w) v = is_max ? fmaxf(v, red[w]) : v + red[w];
  return v;
}

// One block per query: the Gumbel-top-k keys of the policy of Eq. 11 over the
// non-empty groups, key_g = log mu_g - log(-log u_g), with mu_g = eps / |G_t|
// + (1 - eps) softmax(s / tau)_g and u_g the query's Philox uniform for g
// (word g mod 4 of the counter (g / 4, b, offset); top 23 bits plus one half,
// times 2^-23).  The k largest keys are k draws without replacement from
// mu (Kool, van Hoof and Welling, ICML 2019).  Empty groups get -inf.
__global__ void __launch_bounds__(256) policy_keys_kernel(PolicyArgs a) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  __shared__ float red[32];
  const int b = blockIdx.x;
  const int64_t plane = (int64_t)a.B * a.G;
  const float *src = a.s1 + (int64_t)b * a.G;
  float *keys = a.keys + (int64_t)b * a.G;
  // Scores (summed over the planes) into the key row, and their maximum.
  float m = -INFINITY;
  for (int g = threadIdx.x; g < a.G; g += blockDim.x) {
    float s = src[g];
    for (int p = 1; p < a.planes; ++p) s += src[p * plane + g];
    keys[g] = s;
    if (a.count[g] > 0) m = fmaxf(m, s * a.inv_tau);
  }
  m = block_reduce(m, true, red);
  float sum = 0.f;
  for (int g = threadIdx.x; g < a.G; g += blockDim.x) {
    if (a.count[g] > 0) sum += expf(keys[g] * a.inv_tau - m);
  }
  sum = block_reduce(sum, false, red);
  const float lse = m + logf(sum);
  const float log_unif = a.eps > 0.f ? logf(a.eps / (float)a.n_nonempty) : -INFINITY;
  const float log_soft = a.eps < 1.f ? log1pf(-a.eps) : -INFINITY;
  for (int q = threadIdx.x; q * 4 < a.G; q += blockDim.x) {
    const uint4 r = philox4x32_10(make_uint4((uint32_t)q, (uint32_t)b, a.off_lo, a.off_hi), a.key);
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int g = q * 4 + j;
      if (g >= a.G) break;
      if (a.count[g] == 0) {
        keys[g] = -INFINITY;
        continue;
      }
      const float z = keys[g] * a.inv_tau - lse;
      float log_mu;
      if (a.eps == 0.f) {
        log_mu = z;
      } else {
        const float c = log_soft + z;
        const float hi = fmaxf(log_unif, c), lo = fminf(log_unif, c);
        log_mu = hi + log1pf(expf(lo - hi));
      }
      const float u = ((float)(w[j] >> 9) + 0.5f) * (1.0f / 8388608.0f);
      keys[g] = log_mu - logf(-logf(u));
    }
  }
}

// The drawn groups' scores: group_score[b][j] = s[b][group_idx[b][j]]
// (planes summed in order, as the selection sums them), -inf for padding.
__global__ void policy_scores_kernel(const float *__restrict__ s1, int planes, int B, int G, int kg,
                                     const int32_t *__restrict__ group_idx, float *__restrict__ group_score) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * kg) return;
  const int g = group_idx[t];
  const int64_t b = t / kg;
  float s = -INFINITY;
  if (g >= 0) {
    const int64_t plane = (int64_t)B * G;
    s = s1[b * G + g];
    for (int p = 1; p < planes; ++p) s += s1[p * plane + b * G + g];
  }
  group_score[t] = s;
}

// ---------------------------------------------------------------- flat scan

// The ascending list of non-empty groups (one block, 1024 groups per pass).
__global__ void __launch_bounds__(1024) flat_groups_kernel(const int32_t *__restrict__ count, int G,
                                                           int32_t *__restrict__ list) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  __shared__ int warp_n[32];
  __shared__ int base;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) base = 0;
  __syncthreads();
  for (int g0 = 0; g0 < G; g0 += 1024) {
    const int g = g0 + (int)threadIdx.x;
    const bool ne = g < G && count[g] > 0;
    const unsigned bal = __ballot_sync(0xffffffffu, ne);
    if (lane == 0) warp_n[warp] = __popc(bal);
    __syncthreads();
    int before = base;
    for (int w = 0; w < warp; ++w) before += warp_n[w];
    if (ne) list[before + __popc(bal & ((1u << lane) - 1u))] = g;
    __syncthreads();
    if (threadIdx.x == 0) {
      int n = 0;
      for (int w = 0; w < 32; ++w) n += warp_n[w];
      base += n;
    }
    __syncthreads();
  }
}

// Every query selects every non-empty group: group_idx[b][j] = list[j].
__global__ void flat_fill_kernel(const int32_t *__restrict__ list, int64_t rows, int kg,
                                 int32_t *__restrict__ group_idx) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t < rows) group_idx[t] = list[t % kg];
}

// ---------------------------------------------------------------- bucketing

// The bucketing steps are device functions over one row or one group, run
// by a kernel each or, for small batches, all in one block.
__device__ __forceinline__ void bucket_bits_row(int64_t t, const int32_t *__restrict__ gidx, int kg, int W,
                                                uint32_t *bits) {
  const int b = (int)(t / kg);
  const int32_t g = gidx[t];
  if (g >= 0) atomicOr(&bits[(int64_t)g * W + (b >> 5)], 1u << (b & 31));
}

__global__ void bucket_bits_kernel(const int32_t *__restrict__ gidx, int B, int kg, int W,
                                   uint32_t *__restrict__ bits) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t < (int64_t)B * kg) bucket_bits_row(t, gidx, kg, W, bits);
}

// One warp per group: the bucket size c_g and, per bitmap word, how many of
// the group's queries come before it (wpre[g][w]).
__device__ __forceinline__ void bucket_count_group(int g, int lane, const uint32_t *bits, int W,
                                                   int32_t *__restrict__ cnt, int32_t *__restrict__ wpre) {
  int running = 0;
  for (int w0 = 0; w0 < W; w0 += 32) {
    const int w = w0 + lane;
    const int pc = w < W ? __popc(bits[(int64_t)g * W + w]) : 0;
    int incl = pc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(kFullMask, incl, o);
      if (lane >= o) incl += t;
    }
    if (w < W) wpre[(int64_t)g * W + w] = running + incl - pc;
    running += __shfl_sync(kFullMask, incl, 31);
  }
  if (lane == 0) cnt[g] = running;
}

__global__ void bucket_count_kernel(const uint32_t *__restrict__ bits, int G, int W,
                                    int32_t *__restrict__ cnt, int32_t *__restrict__ wpre) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int g = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (g < G) bucket_count_group(g, threadIdx.x & 31, bits, W, cnt, wpre);
}

// pos[b][j] = rank of query b in the bucket of its j-th selected group: the
// group's queries before b's bitmap word plus those before b within it.
__device__ __forceinline__ void bucket_pos_row(int64_t t, const uint32_t *bits, const int32_t *wpre, int W,
                                               const int32_t *__restrict__ gidx, int kg, int32_t *__restrict__ pos) {
  const int g = gidx[t];
  if (g < 0) return;
  const int b = (int)(t / kg);
  const int w = b >> 5;
  const uint32_t below = bits[(int64_t)g * W + w] & ((1u << (b & 31)) - 1u);
  pos[t] = wpre[(int64_t)g * W + w] + __popc(below);
}

__global__ void bucket_pos_kernel(const uint32_t *__restrict__ bits, const int32_t *__restrict__ wpre, int W,
                                  const int32_t *__restrict__ gidx, int64_t rows, int kg,
                                  int32_t *__restrict__ pos) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (t < rows) bucket_pos_row(t, bits, wpre, W, gidx, kg, pos);
}

// Which fine kernel scores a group's bucket: buckets of at least tc_min
// queries go to the tensor-core kernel in chunks of 128 queries and page
// segments of seg_tc pages, smaller ones to the SIMT kernel in chunks of
// qc_simt queries and segments of seg_simt pages.
struct Route {
  int tc_min, qc_simt, seg_simt, seg_tc, pairs;
  __host__ __device__ bool tc(int c) const { return c >= tc_min; }
  // Tensor-core buckets of more than one chunk run on SM pairs (when on).
  __host__ __device__ bool pair(int c) const { return pairs && tc(c) && c > kTcRows; }
  __host__ __device__ int qc(int c) const { return tc(c) ? kTcRows : qc_simt; }
  __host__ __device__ int seg(int c) const { return tc(c) ? seg_tc : seg_simt; }
  __host__ __device__ int nseg(int c, int pages) const { return (pages + seg(c) - 1) / seg(c); }
  // Work units of a group: (chunk, segment) pairs, or (chunk pair, segment)
  // pairs on SM pairs.
  __host__ __device__ int64_t units(int c, int pages) const {
    if (c <= 0) return 0;
    const int64_t nch = (c + qc(c) - 1) / qc(c);
    return (pair(c) ? (nch + 1) / 2 : nch) * nseg(c, pages);
  }
  // Tensor-core tiles (two pages each) of a group: every chunk of the bucket
  // against every page pair.
  __host__ __device__ int64_t tc_tiles(int c, int pages) const {
    return tc(c) ? (int64_t)((c + kTcRows - 1) / kTcRows) * ((pages + 1) / 2) : 0;
  }
};

// Pages per tensor-core unit: the smallest power of two whose tiles (two
// pages each) are at least half the tiles per SM, within [kTcSegPagesMin,
// kTcSegPagesMax].  Long segments mean fewer cold top-k lists and fewer
// partial records; short ones keep every SM busy when the tensor-core work
// is small (units are taken dynamically, so a few long ones balance out).
constexpr int kTcSegPagesMin = 4;
constexpr int kTcSegPagesMax = 256;
__device__ __forceinline__ int tc_seg_pages(int64_t tiles, int sms) {
  int seg = kTcSegPagesMin;
  while (seg < kTcSegPagesMax && (int64_t)seg * sms <= tiles) seg *= 2;  // seg/2 tiles <= tiles per SM
  return seg;
}

// Single block: chooses the pages per tensor-core unit from the total
// tensor-core tiles (written to seg_tc_dev), then per group the bucket size
// c_g, its work units (in the SIMT, one-SM or SM-pair tensor-core list) and
// its partial records c_g * nseg_g, with exclusive scans over the groups
// (warp shuffles, then one pass over the 32 warp totals).
// n_units = {SIMT units, one-SM tensor-core units, SM-pair units}.
__device__ void bucket_scan_block(
    const int32_t *__restrict__ cnt, const int32_t *__restrict__ page_off, int G, Route rt, int sms,
    int32_t *__restrict__ bucket_off, int32_t *__restrict__ unit_off, int32_t *__restrict__ unit_off_tc,
    int32_t *__restrict__ unit_off_tc2, int64_t *__restrict__ part_off, int32_t *__restrict__ n_units,
    int32_t *__restrict__ seg_tc_dev) {
  constexpr int kVals = 5;  // bucket rows, SIMT units, one-SM units, records, SM-pair units
  __shared__ int64_t wsum[kVals][32];
  __shared__ int64_t tiles_sh;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (G + 1023) / 1024;
  const int lo = min(G, tid * per), hi = min(G, lo + per);
  {
    int64_t x = 0;
    for (int g = lo; g < hi; ++g) x += rt.tc_tiles(cnt[g], page_off[g + 1] - page_off[g]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(kFullMask, x, o);
    if (lane == 0) wsum[0][warp] = x;
    __syncthreads();
    if (tid == 0) {
      int64_t t = 0;
      for (int w = 0; w < 32; ++w) t += wsum[0][w];
      tiles_sh = t;
    }
    __syncthreads();
    rt.seg_tc = tc_seg_pages(tiles_sh, sms);
    if (tid == 0) *seg_tc_dev = rt.seg_tc;
  }
  int64_t v[kVals] = {0, 0, 0, 0, 0};
  auto add = [&](int64_t (&acc)[kVals], int g) {
    const int c = cnt[g], pages = page_off[g + 1] - page_off[g];
    const int64_t u = rt.units(c, pages);
    const bool pr = rt.pair(c), tc = rt.tc(c);
    acc[0] += c;
    acc[1] += tc ? 0 : u;
    acc[2] += tc && !pr ? u : 0;
    acc[3] += (int64_t)c * rt.nseg(c, pages);
    acc[4] += pr ? u : 0;
  };
  for (int g = lo; g < hi; ++g) add(v, g);
  // Inclusive scan within the warp, then the warp totals.
  int64_t incl[kVals];
#pragma unroll
  for (int i = 0; i < kVals; ++i) {
    incl[i] = v[i];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t t = __shfl_up_sync(kFullMask, incl[i], o);
      if (lane >= o) incl[i] += t;
    }
  }
  __syncthreads();  // wsum[0] was read above
  if (lane == 31) {
#pragma unroll
    for (int i = 0; i < kVals; ++i) wsum[i][warp] = incl[i];
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int i = 0; i < kVals; ++i) {
      int64_t x = wsum[i][lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int64_t t = __shfl_up_sync(kFullMask, x, o);
        if (lane >= o) x += t;
      }
      wsum[i][lane] = x;  // inclusive over warps
    }
  }
  __syncthreads();
  int64_t run[kVals];
#pragma unroll
  for (int i = 0; i < kVals; ++i) run[i] = (warp > 0 ? wsum[i][warp - 1] : 0) + incl[i] - v[i];
  for (int g = lo; g < hi; ++g) {
    bucket_off[g] = (int32_t)run[0];
    unit_off[g] = (int32_t)run[1];
    unit_off_tc[g] = (int32_t)run[2];
    part_off[g] = run[3];
    unit_off_tc2[g] = (int32_t)run[4];
    add(run, g);
  }
  if (tid == 1023) {
    bucket_off[G] = (int32_t)run[0];
    unit_off[G] = (int32_t)run[1];
    unit_off_tc[G] = (int32_t)run[2];
    part_off[G] = run[3];
    unit_off_tc2[G] = (int32_t)run[4];
    n_units[0] = (int32_t)run[1];
    n_units[1] = (int32_t)run[2];
    n_units[2] = (int32_t)run[4];
  }
}

__global__ void __launch_bounds__(1024) bucket_scan_kernel(
    const int32_t *__restrict__ cnt, const int32_t *__restrict__ page_off, int G, Route rt, int sms,
    int32_t *__restrict__ bucket_off, int32_t *__restrict__ unit_off, int32_t *__restrict__ unit_off_tc,
    int32_t *__restrict__ unit_off_tc2, int64_t *__restrict__ part_off, int32_t *__restrict__ n_units,
    int32_t *__restrict__ seg_tc_dev) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  bucket_scan_block(cnt, page_off, G, rt, sms, bucket_off, unit_off, unit_off_tc, unit_off_tc2, part_off, n_units,
                    seg_tc_dev);
}

__device__ __forceinline__ void bucket_fill_group(int g, int lane, uint32_t *bits, bool clear, int W,
                                                  const int32_t *__restrict__ bucket_off,
                                                  const int32_t *__restrict__ cnt,
                                                  const int32_t *__restrict__ page_off, const Route &rt,
                                                  const int32_t *__restrict__ unit_off,
                                                  const int32_t *__restrict__ unit_off_tc,
                                                  const int32_t *__restrict__ unit_off_tc2,
                                                  int32_t *__restrict__ bucket, int32_t *__restrict__ bucket_group,
                                                  int4 *__restrict__ units, int4 *__restrict__ units_tc,
                                                  int4 *__restrict__ units_tc2) {
  int running = 0;
  const int base = bucket_off[g];
  for (int w0 = 0; w0 < W; w0 += 32) {
    uint32_t word = w0 + lane < W ? bits[(int64_t)g * W + w0 + lane] : 0u;
    // The global bitmap of the multi-kernel bucketing is zero between
    // queries: read here for the last time, so cleared for the next query.
    // (The one-block bucketing's bitmap is in shared memory, where other
    // threads may still be reading it.)
    if (clear && w0 + lane < W) bits[(int64_t)g * W + w0 + lane] = 0u;
    int pc = __popc(word), incl = pc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int t = __shfl_up_sync(kFullMask, incl, o);
      if (lane >= o) incl += t;
    }
    int r = running + incl - pc;
    while (word) {
      int bit = __ffs(word) - 1;
      word &= word - 1;
      int b = (w0 + lane) * 32 + bit;
      bucket[base + r] = b;
      bucket_group[base + r] = g;
      ++r;
    }
    running += __shfl_sync(kFullMask, incl, 31);
  }
  int c = cnt[g];
  if (c == 0) return;
  const int pages = page_off[g + 1] - page_off[g];
  const int nseg = rt.nseg(c, pages);
  const int n_u = (int)rt.units(c, pages);
  // (group, chunk or chunk pair, segment)
  int4 *dst = rt.pair(c) ? units_tc2 + unit_off_tc2[g] : rt.tc(c) ? units_tc + unit_off_tc[g] : units + unit_off[g];
  for (int u = lane; u < n_u; u += 32) dst[u] = make_int4(g, u / nseg, u % nseg, 0);
}

// One warp per group: bucket[g] lists its queries in increasing order.
// Also writes the group's work units (group, chunk, segment) to the list of
// the kernel that will score them, and the group of every bucket row.
__global__ void bucket_fill_kernel(uint32_t *__restrict__ bits, int G, int W,
                                   const int32_t *__restrict__ bucket_off,
                                   const int32_t *__restrict__ cnt,
                                   const int32_t *__restrict__ page_off, Route rt,
                                   const int32_t *__restrict__ seg_tc_dev,
                                   const int32_t *__restrict__ unit_off,
                                   const int32_t *__restrict__ unit_off_tc,
                                   const int32_t *__restrict__ unit_off_tc2,
                                   int32_t *__restrict__ bucket, int32_t *__restrict__ bucket_group,
                                   int4 *__restrict__ units,
                                   int4 *__restrict__ units_tc,
                                   int4 *__restrict__ units_tc2,
                                   unsigned *__restrict__ thr_zero, int thr_words,
                                   int32_t *__restrict__ ctr_zero) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  // Also clears the tensor-core kernel's shared bounds and unit counters
  // (when given), which no earlier kernel of the query touches.
  if (thr_zero) {
    const int64_t t0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    for (int64_t t = t0; t < thr_words; t += (int64_t)gridDim.x * blockDim.x) thr_zero[t] = 0u;
    if (t0 < 2) ctr_zero[t0] = 0;
  }
  const int g = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  rt.seg_tc = *seg_tc_dev;
  if (g < G) {
    bucket_fill_group(g, threadIdx.x & 31, bits, true, W, bucket_off, cnt, page_off, rt, unit_off, unit_off_tc,
                      unit_off_tc2, bucket, bucket_group, units, units_tc, units_tc2);
  }
}

// The whole bucketing in one block for small batches (the bitmap in shared
// memory): the steps of the kernels above in order, a block barrier between
// them, one launch instead of five plus a memset.
struct BucketSmallArgs {
  const int32_t *gidx;
  int B, kg, G, W;
  const int32_t *page_off;
  Route rt;
  int sms;
  int32_t *cnt, *wpre, *pos, *bucket_off, *unit_off, *unit_off_tc, *unit_off_tc2;
  int64_t *part_off;
  int32_t *n_units, *seg_tc_dev, *bucket, *bucket_group;
  int4 *units, *units_tc, *units_tc2;
  unsigned *thr_zero;
  int thr_words;  // words of thr_zero
  int32_t *ctr_zero;
};
// One block pays off only for small problems: with programmatic dependent
// launch the five kernels already win on the 65k workload (256 groups x 8
// words, 2,048 rows: 20 us against 28 us), while the 8-query one (32 rows)
// still saves launches in one block.
constexpr int kBucketSmallWords = 4096;  // bitmap words held in shared memory (16 KiB)
constexpr int64_t kBucketSmallRows = 1024;

__global__ void __launch_bounds__(1024) bucket_small_kernel(BucketSmallArgs a) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  extern __shared__ uint32_t sbits[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t rows = (int64_t)a.B * a.kg;
  const int words = a.G * a.W;
  for (int i = tid; i < words; i += 1024) sbits[i] = 0u;
  if (a.thr_zero) {
    for (int i = tid; i < a.thr_words; i += 1024) a.thr_zero[i] = 0u;
    if (tid < 2) a.ctr_zero[tid] = 0;
  }
  __syncthreads();
  for (int64_t t = tid; t < rows; t += 1024) bucket_bits_row(t, a.gidx, a.kg, a.W, sbits);
  __syncthreads();
  for (int g = warp; g < a.G; g += 32) bucket_count_group(g, lane, sbits, a.W, a.cnt, a.wpre);
  __syncthreads();  // counts and word prefixes (global) visible to the block
  bucket_scan_block(a.cnt, a.page_off, a.G, a.rt, a.sms, a.bucket_off, a.unit_off, a.unit_off_tc, a.unit_off_tc2,
                    a.part_off, a.n_units, a.seg_tc_dev);
  __syncthreads();
  Route rt = a.rt;
  rt.seg_tc = *a.seg_tc_dev;
  for (int64_t t = tid; t < rows; t += 1024) bucket_pos_row(t, sbits, a.wpre, a.W, a.gidx, a.kg, a.pos);
  for (int g = warp; g < a.G; g += 32) {
    bucket_fill_group(g, lane, sbits, false, a.W, a.bucket_off, a.cnt, a.page_off, rt, a.unit_off, a.unit_off_tc,
                      a.unit_off_tc2, a.bucket, a.bucket_group, a.units, a.units_tc, a.units_tc2);
  }
}


// ------------------------------------------------------------ fine (SIMT)

struct FineArgs {
  const void *pool;
  int d;
  const int32_t *slot_id;
  const int32_t *page_list;
  const int32_t *page_off;
  const int32_t *count;
  const void *Q;
  const int32_t *bucket;
  const int32_t *bucket_off;
  const int32_t *cnt;
  const int4 *units;
  const int32_t *n_units;
  const int64_t *part_off;
  int ke;
  float inv_tau;
  int seg_pages;
  float2 *part_ml;
  float *part_s;
  int32_t *part_id;
};

constexpr int kFineWarps = 8;

// 16 bytes of entry data as fp32 values.
template <typename T>
struct Unpack;
template <>
struct Unpack<__nv_bfloat16> {
  static constexpr int kN = 8;
  __device__ static void run(const uint4 &w, float *f) {
    f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
    f[4] = bf16lo(w.z); f[5] = bf16hi(w.z); f[6] = bf16lo(w.w); f[7] = bf16hi(w.w);
  }
};
template <>
struct Unpack<float> {
  static constexpr int kN = 4;
  __device__ static void run(const uint4 &w, float *f) {
    f[0] = __uint_as_float(w.x); f[1] = __uint_as_float(w.y);
    f[2] = __uint_as_float(w.z); f[3] = __uint_as_float(w.w);
  }
};

// Work unit = (group g, bucket chunk c, page segment s): the up-to-QC queries
// bucket[g][c*QC ...] against the rows of pages [s*seg, (s+1)*seg) of g.
// Each warp streams rows (coalesced 16-byte loads), reduces the dot products
// with shuffles and keeps, per query, the online softmax state (max, sum of
// exp) and a warp-distributed top-k; the warps are merged in shared memory
// and one partial record per (query, unit) is written.
template <typename T, int QC, int B>
__global__ void __launch_bounds__(kFineWarps * 32, 2) fine_simt_kernel(FineArgs a) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  extern __shared__ __align__(16) unsigned char smem_raw[];
  constexpr int kN = Unpack<T>::kN;
  const int d = a.d;
  float *qs = reinterpret_cast<float *>(smem_raw);              // [QC][d]
  float *ws = qs + QC * d;                                       // [warps][QC][64]
  int *wi = reinterpret_cast<int *>(ws + kFineWarps * QC * 64);  // [warps][QC][64]
  float *wm = reinterpret_cast<float *>(wi + kFineWarps * QC * 64);  // [warps][QC]
  float *wl = wm + kFineWarps * QC;                                   // [warps][QC]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_vec = d / kN;  // 16-byte vectors per row
  const int ke = a.ke;
  const int n_units = *a.n_units;
  const uint4 *pool = static_cast<const uint4 *>(a.pool);
  const T *Q = static_cast<const T *>(a.Q);

  for (int u = blockIdx.x; u < n_units; u += gridDim.x) {
    const int4 U = a.units[u];
    const int g = U.x, c = U.y, s = U.z;
    const int cg = a.cnt[g];
    const int q0 = c * QC;
    const int nq = min(QC, cg - q0);
    const int *bq = a.bucket + a.bucket_off[g] + q0;

    __syncthreads();  // the previous unit is done with shared memory
    for (int i = tid; i < nq * (d / 4); i += blockDim.x) {
      int j = i / (d / 4), k = (i % (d / 4)) * 4;
      const T *src = Q + (int64_t)bq[j] * d + k;
      float4 v;
      if constexpr (sizeof(T) == 2) {
        uint2 w = *reinterpret_cast<const uint2 *>(src);
        v = make_float4(bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y));
      } else {
        v = *reinterpret_cast<const float4 *>(src);
      }
      *reinterpret_cast<float4 *>(qs + j * d + k) = v;
    }
    __syncthreads();

    const int pg0 = a.page_off[g];
    const int npages = a.page_off[g + 1] - pg0;
    const int p_beg = s * a.seg_pages;
    const int p_end = min(npages, p_beg + a.seg_pages);
    const int r0 = p_beg * kPageRows;
    const int r1 = min(p_end * kPageRows, a.count[g]);

    float m[QC], l[QC], ts[QC];
    int ti[QC];
    WarpList lst[QC];
#pragma unroll
    for (int j = 0; j < QC; ++j) {
      m[j] = -INFINITY;
      l[j] = 0.f;
      ts[j] = -INFINITY;
      ti[j] = INT_MAX;
      lst[j].init();
    }

    for (int r = r0 + warp; r < r1; r += kFineWarps) {
      const int64_t slot = (int64_t)a.page_list[pg0 + r / kPageRows] * kPageRows + (r % kPageRows);
      const int id = a.slot_id[slot];
      const uint4 *row = pool + slot * n_vec;
      float acc[QC];
#pragma unroll
      for (int j = 0; j < QC; ++j) acc[j] = 0.f;
      // B 16-byte loads per lane are issued before any is used, so each warp
      // keeps B * 512 bytes of the row in flight.
      for (int v0 = lane; v0 < n_vec; v0 += 32 * B) {
        uint4 w[B];
#pragma unroll
        for (int i = 0; i < B; ++i) {
          const int v = v0 + 32 * i;
          w[i] = v < n_vec ? row[v] : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int i = 0; i < B; ++i) {
          const int v = v0 + 32 * i;
          if (v >= n_vec) break;
          float f[kN];
          Unpack<T>::run(w[i], f);
#pragma unroll
          for (int j = 0; j < QC; ++j) {
            if (j < nq) {
              const float *q = qs + j * d + v * kN;
#pragma unroll
              for (int t = 0; t < kN; t += 4) {
                float4 qq = *reinterpret_cast<const float4 *>(q + t);
                acc[j] = fmaf(f[t], qq.x, acc[j]);
                acc[j] = fmaf(f[t + 1], qq.y, acc[j]);
                acc[j] = fmaf(f[t + 2], qq.z, acc[j]);
                acc[j] = fmaf(f[t + 3], qq.w, acc[j]);
              }
            }
          }
        }
      }
#pragma unroll
      for (int j = 0; j < QC; ++j) {
        if (j < nq) {
          float sc = warp_sum(acc[j]);
          float z = sc * a.inv_tau;
          if (z > m[j]) {
            l[j] = l[j] * expf(m[j] - z) + 1.f;
            m[j] = z;
          } else {
            l[j] += expf(z - m[j]);
          }
          if (better(sc, id, ts[j], ti[j])) {
            lst[j].insert(ke, sc, id);
            lst[j].kth(ke, ts[j], ti[j]);
          }
        }
      }
    }

    // Hand each warp's state to shared memory, then warp j merges query j.
#pragma unroll
    for (int j = 0; j < QC; ++j) {
      if (j < nq) {
        int o = (warp * QC + j) * 64;
        ws[o + lane] = lst[j].s0;
        wi[o + lane] = lst[j].i0;
        ws[o + 32 + lane] = lst[j].s1;
        wi[o + 32 + lane] = lst[j].i1;
        if (lane == 0) {
          wm[warp * QC + j] = m[j];
          wl[warp * QC + j] = l[j];
        }
      }
    }
    __syncthreads();
    for (int j = warp; j < nq; j += kFineWarps) {
      float M = -INFINITY;
      for (int w = 0; w < kFineWarps; ++w) M = fmaxf(M, wm[w * QC + j]);
      float Ls = 0.f;
      for (int w = 0; w < kFineWarps; ++w) {
        float mw = wm[w * QC + j];
        if (mw != -INFINITY) Ls += wl[w * QC + j] * expf(mw - M);
      }
      WarpList F;
      F.init();
      float fs = -INFINITY;
      int fi = INT_MAX;
      for (int w = 0; w < kFineWarps; ++w) {
        for (int h = 0; h < 2; ++h) {
          if (h * 32 >= ke) break;
          int o = (w * QC + j) * 64 + h * 32;
          float cs = ws[o + lane];
          int ci = wi[o + lane];
          unsigned mask = __ballot_sync(kFullMask, h * 32 + lane < ke && ci != INT_MAX && better(cs, ci, fs, fi));
          while (mask) {
            int src = __ffs(mask) - 1;
            mask &= mask - 1;
            float vs = __shfl_sync(kFullMask, cs, src);
            int vi = __shfl_sync(kFullMask, ci, src);
            F.insert(ke, vs, vi);
            F.kth(ke, fs, fi);
          }
        }
      }
      const int64_t pidx = a.part_off[g] + (int64_t)s * cg + q0 + j;
      if (lane == 0) a.part_ml[pidx] = make_float2(M, Ls);
      if (lane < ke) {
        a.part_s[pidx * ke + lane] = F.s0;
        a.part_id[pidx * ke + lane] = F.i0;
      }
      if (lane + 32 < ke) {
        a.part_s[pidx * ke + lane + 32] = F.s1;
        a.part_id[pidx * ke + lane + 32] = F.i1;
      }
    }
  }
}

// ------------------------------------------------------------------- merge

struct MergeArgs {
  const int32_t *gidx;
  int B, kg, ke;
  const int32_t *count;
  const int32_t *pos;
  const int32_t *cnt;
  const int32_t *page_off;
  Route rt;                  // seg_tc is replaced by *seg_tc_dev
  const int32_t *seg_tc_dev;
  const int64_t *part_off;
  const float2 *part_ml;
  const float *part_s;
  const int32_t *part_id;
  float inv_tau, eps;
  int32_t *entry_idx;
  float *entry_score, *entry_weight, *lse;
};

// A team of WPQ warps per query (8 warps per block): combine its partial
// records (one per selected group and page segment) -- log-sum-exp of the
// softmax statistics and the final top-k.  Warp w of a team takes the
// selected groups j = w, w + WPQ, ...; the team's first warp then combines
// the team's statistics and lists.
constexpr int kMergeWarps = 8;

template <int WPQ>
__global__ void __launch_bounds__(kMergeWarps * 32, 1) merge_kernel(MergeArgs a) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  __shared__ float ls[kMergeWarps][64];
  __shared__ int li[kMergeWarps][64];
  __shared__ float wM[kMergeWarps], wL[kMergeWarps];
  __shared__ long long wN[kMergeWarps];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * (kMergeWarps / WPQ) + warp / WPQ;
  const int sw = warp % WPQ;
  const bool live = b < a.B;  // uniform per warp
  const int ke = a.ke;
  float M = -INFINITY, L = 0.f;
  int64_t nb = 0;
  WarpList F;
  F.init();
  float fs = -INFINITY;
  int fi = INT_MAX;
  auto offer = [&](float cs, int ci, int limit) {
    unsigned mask = __ballot_sync(kFullMask, lane < limit && ci != INT_MAX && better(cs, ci, fs, fi));
    while (mask) {
      const int src = __ffs(mask) - 1;
      mask &= mask - 1;
      F.insert(ke, __shfl_sync(kFullMask, cs, src), __shfl_sync(kFullMask, ci, src));
      F.kth(ke, fs, fi);
    }
  };
  // Takes in a sorted list of ke <= 32 pairs held one per lane (padding past
  // ke): skipped when its best pair cannot enter the top-ke, else merged.
  auto take32 = [&](float cs, int ci) {
    const float bs = __shfl_sync(kFullMask, cs, 0);
    const int bi = __shfl_sync(kFullMask, ci, 0);
    if (bi != INT_MAX && better(bs, bi, fs, fi)) {
      F.merge32(cs, ci);
      F.kth(ke, fs, fi);
    }
  };
  // The index data of this warp's groups j = sw + t * WPQ, loaded by lane
  // t % 32 (slot t / 32) in parallel, then handed round by shuffles.
  struct GroupRecs {
    int g, p, cg, nseg;
    long long base;
  };
  Route rt = a.rt;
  rt.seg_tc = *a.seg_tc_dev;
  auto load_group = [&](int t) {
    GroupRecs r{-1, 0, 0, 0, 0};
    const int j = sw + t * WPQ;
    if (live && j < a.kg) {
      r.g = a.gidx[(int64_t)b * a.kg + j];
      if (r.g >= 0) {
        r.p = a.pos[(int64_t)b * a.kg + j];
        r.cg = a.cnt[r.g];
        r.nseg = rt.nseg(r.cg, a.page_off[r.g + 1] - a.page_off[r.g]);
        r.base = a.part_off[r.g];
        nb += a.count[r.g];
      }
    }
    return r;
  };
  // Records are taken 32 at a time, one per lane, across group boundaries:
  // each lane reads its record's softmax statistics and best pair, the
  // statistics are combined by warp reductions, and only records whose best
  // pair can still enter the top-ke are read in full (up to 4 at a time).
  const int n_t = live ? (a.kg - sw + WPQ - 1) / WPQ : 0;
  for (int t0 = 0; t0 < n_t; t0 += 32) {
    const GroupRecs gr = load_group(t0 + lane);
    const int nseg = gr.g >= 0 ? gr.nseg : 0;
    int incl = nseg;  // inclusive prefix of the records over the lanes' groups
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(kFullMask, incl, o);
      if (lane >= o) incl += v;
    }
    const int excl = incl - nseg;
    const int total = __shfl_sync(kFullMask, incl, 31);
    for (int r0 = 0; r0 < total; r0 += 32) {
      const int r = r0 + lane;
      // The lane whose group holds record r: the last lane with excl <= r.
      int own = 0;
#pragma unroll
      for (int step = 16; step > 0; step >>= 1) {
        if (__shfl_sync(kFullMask, excl, own + step) <= r) own += step;
      }
      const int seg = r - __shfl_sync(kFullMask, excl, own);
      const int p = __shfl_sync(kFullMask, gr.p, own);
      const int cg = __shfl_sync(kFullMask, gr.cg, own);
      const long long base = __shfl_sync(kFullMask, gr.base, own);
      const bool valid = r < total;
      const long long pidx = base + (long long)seg * cg + p;
      const float2 ml = valid ? a.part_ml[pidx] : make_float2(-INFINITY, 0.f);
      const float hs = valid ? a.part_s[pidx * ke] : -INFINITY;
      const int hi = valid ? a.part_id[pidx * ke] : INT_MAX;
      const float Mb = warp_max(ml.x);
      if (Mb != -INFINITY) {
        const float Lb = warp_sum(ml.x == -INFINITY ? 0.f : ml.y * expf(ml.x - Mb));
        const float Mn = fmaxf(M, Mb);
        L = L * expf(M - Mn) + Lb * expf(Mb - Mn);
        M = Mn;
      }
      unsigned todo = __ballot_sync(kFullMask, hi != INT_MAX && better(hs, hi, fs, fi));
      while (todo) {
        constexpr int kTake = 4;
        int src[kTake];
#pragma unroll
        for (int i = 0; i < kTake; ++i) {
          src[i] = todo ? __ffs(todo) - 1 : -1;
          if (todo) todo &= todo - 1;
        }
        float cs[kTake][2];
        int ci[kTake][2];
#pragma unroll
        for (int i = 0; i < kTake; ++i) {
          const long long q = __shfl_sync(kFullMask, pidx, src[i] < 0 ? 0 : src[i]);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int tt = h * 32 + lane;
            const bool in = src[i] >= 0 && tt < ke;
            cs[i][h] = in ? a.part_s[q * ke + tt] : -INFINITY;
            ci[i][h] = in ? a.part_id[q * ke + tt] : INT_MAX;
          }
        }
#pragma unroll
        for (int i = 0; i < kTake; ++i) {
          if (src[i] < 0) break;  // uniform
          if (ke <= 32) {
            take32(cs[i][0], ci[i][0]);
          } else {
#pragma unroll
            for (int h = 0; h < 2; ++h) offer(cs[i][h], ci[i][h], ke - h * 32);
          }
        }
        // Drop the records the raised k-th best now excludes.
        todo &= __ballot_sync(kFullMask, hi != INT_MAX && better(hs, hi, fs, fi));
      }
    }
  }
  // Entries behind this warp's groups (each lane counted its own groups).
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) nb += __shfl_xor_sync(kFullMask, nb, o);
  if constexpr (WPQ > 1) {
    ls[warp][lane] = F.s0;
    li[warp][lane] = F.i0;
    ls[warp][lane + 32] = F.s1;
    li[warp][lane + 32] = F.i1;
    if (lane == 0) {
      wM[warp] = M;
      wL[warp] = L;
      wN[warp] = nb;
    }
    __syncthreads();
    if (sw != 0 || !live) return;
    M = -INFINITY;
    L = 0.f;
    nb = 0;
    for (int w = warp; w < warp + WPQ; ++w) {
      nb += wN[w];
      if (wM[w] != -INFINITY) {
        const float Mn = fmaxf(M, wM[w]);
        L = L * expf(M - Mn) + wL[w] * expf(wM[w] - Mn);
        M = Mn;
      }
    }
    F.init();
    fs = -INFINITY;
    fi = INT_MAX;
    for (int w = warp; w < warp + WPQ; ++w) {
      if (ke <= 32) {
        take32(ls[w][lane], li[w][lane]);
      } else {
        for (int h = 0; h * 32 < ke; ++h) offer(ls[w][h * 32 + lane], li[w][h * 32 + lane], ke - h * 32);
      }
    }
  }
  if (!live) return;
  const float lse_b = nb > 0 ? M + logf(L) : -INFINITY;
  const float unif = nb > 0 ? a.eps / (float)nb : 0.f;
  auto emit = [&](int t, float s, int id) {
    int64_t o = (int64_t)b * ke + t;
    if (id == INT_MAX) {
      a.entry_idx[o] = -1;
      a.entry_score[o] = -INFINITY;
      a.entry_weight[o] = 0.f;
    } else {
      a.entry_idx[o] = id;
      a.entry_score[o] = s;
      a.entry_weight[o] = unif + (1.f - a.eps) * expf(s * a.inv_tau - lse_b);
    }
  };
  if (lane < ke) emit(lane, F.s0, F.i0);
  if (lane + 32 < ke) emit(lane + 32, F.s1, F.i1);
  if (a.lse && lane == 0) a.lse[b] = lse_b;
}

template <typename T, int QC, int B>
htam_status launch_fine_simt(const FineArgs &fa, int sm_count, int64_t max_units, cudaStream_t st) {
  const int d = fa.d;
  size_t smem = sizeof(float) * QC * d + (sizeof(float) + sizeof(int)) * kFineWarps * QC * 64 +
                sizeof(float) * 2 * kFineWarps * QC;
  auto kernel = fine_simt_kernel<T, QC, B>;
  HTAM_CK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  int per_sm = 0;
  HTAM_CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kFineWarps * 32, smem));
  per_sm = std::max(per_sm, 1);
  int64_t grid = std::min<int64_t>(max_units, (int64_t)sm_count * per_sm);
  if (grid <= 0) return HTAM_OK;
  launch_kernel(kernel, (unsigned)grid, kFineWarps * 32, smem, st, fa);
  HTAM_CK_LAUNCH("fine_simt_kernel");
  return HTAM_OK;
}

// Loads in flight per lane: enough 16-byte vectors for one row, at most
// 32 / QC (so that two blocks of 256 threads fit an SM's registers).
template <typename T, int QC>
htam_status dispatch_batch(const FineArgs &fa, int sm_count, int64_t max_units, cudaStream_t st) {
  const int per_lane = (int)ceil_div((int64_t)fa.d * (int)sizeof(T) / 16, 32);
  if constexpr (QC <= 2) {
    if (per_lane >= 16) return launch_fine_simt<T, QC, 16>(fa, sm_count, max_units, st);
  }
  if constexpr (QC <= 4) {
    if (per_lane > 4) return launch_fine_simt<T, QC, 8>(fa, sm_count, max_units, st);
  }
  if (per_lane > 2) return launch_fine_simt<T, QC, 4>(fa, sm_count, max_units, st);
  if (per_lane > 1) return launch_fine_simt<T, QC, 2>(fa, sm_count, max_units, st);
  return launch_fine_simt<T, QC, 1>(fa, sm_count, max_units, st);
}

template <typename T>
htam_status dispatch_fine_simt(int qc, const FineArgs &fa, int sm_count, int64_t max_units, cudaStream_t st) {
  switch (qc) {
    case 8: return dispatch_batch<T, 8>(fa, sm_count, max_units, st);
    case 4: return dispatch_batch<T, 4>(fa, sm_count, max_units, st);
    case 2: return dispatch_batch<T, 2>(fa, sm_count, max_units, st);
    default: return dispatch_batch<T, 1>(fa, sm_count, max_units, st);
  }
}

}  // namespace

// Queries per CUDA-core work unit: qc * d <= 8192 (at most 8), which keeps
// the staged fp32 query block within 32 KiB and leaves the direct-load
// kernel registers for a long row's loads in flight.
static int simt_query_chunk(int d) {
  int qc = 8;
  while (qc > 1 && (size_t)qc * d > 8192) qc >>= 1;
  return qc;
}

constexpr int kSimtSegPages = 4;

constexpr uint32_t kMaxPolls = 1u << 24;

htam_status query_impl(htam_memory *m, const void *queries, int32_t B, const htam_query_params &p,
                       int32_t *group_idx, float *group_score, int32_t *entry_idx,
                       float *entry_score, float *entry_weight, float *lse, cudaStream_t st,
                       const EdgeRoute *er, bool flat, const SampleSpec *smp) {
  if (B == 0) return HTAM_OK;
  PdlScope pdl(m->pdl != 0);
  // The host mirror of the group sizes bounds the scratch below; the flat
  // scan and the policy draws need the exact non-empty groups, so they wait
  // for the mirror of the last append (the others take the newest one that
  // has landed and bound the rows queued since).
  htam_status s = refresh_mirror(m, flat || smp);
  if (s != HTAM_OK) return s;
  m->n_queries += 1;
  PhaseMark mark(m, st);
  // The flat scan selects every non-empty group (at least one slot, -1 when
  // the memory is empty); the group lists then live in the scratch.
  int n_nonempty = 0;
  if (flat || smp) {
    for (int64_t c : m->h_count) n_nonempty += c > 0;
  }
  const int G = m->n_groups, d = m->d, kg = flat ? std::max(1, n_nonempty) : p.k_groups, ke = p.k_entries;
  const int qc = simt_query_chunk(d);
  // The tensor-core path takes bf16 memories and k_entries <= 32.
  const bool tc_ok = m->dtype == HTAM_BF16 && ke <= kTcMaxK && m->tc_min <= B;
  // seg_tc here is the shortest tensor-core segment (for the bounds below);
  // the kernels take the one bucket_scan_kernel chooses.
  const Route rt{tc_ok ? m->tc_min : INT_MAX, qc, kSimtSegPages, kTcSegPagesMin, m->tc_pairs};

  // Upper bound of the partial records: every query in the buckets of the
  // k_g groups with the most page segments (counted with the shorter
  // segments of the two kernels).  Rows queued after the mirror add at most
  // pending/128 + k_g pages to any k_g groups, so at most
  // (pending/128 + k_g)/seg_min + k_g segments.
  const int seg_min = std::min(kSimtSegPages, kTcSegPagesMin);
  std::vector<int64_t> nseg(G);
  for (int g = 0; g < G; ++g) nseg[g] = ceil_div(ceil_div(m->h_count[g], kPageRows), seg_min);
  std::nth_element(nseg.begin(), nseg.begin() + (kg - 1), nseg.end(), std::greater<int64_t>());
  int64_t seg_sum = 0;
  for (int i = 0; i < kg; ++i) seg_sum += nseg[i];
  if (m->rows_pending > 0) seg_sum += ceil_div(ceil_div(m->rows_pending, kPageRows) + kg, seg_min) + kg;
  const int64_t max_parts = std::max<int64_t>(1, (int64_t)B * seg_sum);
  const int64_t max_units = max_parts;
  const int64_t rows = (int64_t)B * kg;  // bucket rows
  const int W = (int)ceil_div(B, 32);
  // The tensor-core kernel's A rows.  The flat scan's buckets hold every
  // query in order, so TMA reads the query matrix itself.  Otherwise, for
  // batches of up to 2,048 queries of up to 1,024 dims on one-SM units, a
  // copier warp of the kernel copies them from the query matrix (no
  // bucket-ordered copy: 65k workload 0.113 -> 0.110 ms, stream 0.341 ->
  // 0.335 ms); larger batches, longer rows and SM pairs read a
  // bucket-ordered copy by TMA (the copier's 32 copies a lane per K slice
  // made the 4,096-query 1M workload's kernel 0.657 -> 0.797 ms).
  const bool tc_pairs_run = tc_ok && rt.pairs && B > kTcRows;
  const bool a_rows = tc_ok && !flat && !tc_pairs_run && B <= 2048 && d <= 1024;
  const bool q_gather = tc_ok && !flat && !a_rows;
  const size_t qg_bytes = q_gather ? sizeof(__nv_bfloat16) * (size_t)rows * d : 0;

  // Coarse scores: one plane per K split of the tensor-core kernel.
  const int planes = flat ? 0 : m->dtype == HTAM_BF16 && !er ? coarse_tc_splits(B, d, G, m->sm_count) : 1;
  // Edge routing: form the whole utility table once when the batch references
  // more prefix rows than the table has.
  const bool edge_table = er && (int64_t)B * er->P > G;
  const int wpq = warps_per_query(B, m->sm_count);  // warps per query in top-k and merge
  size_t need = Carver::round(sizeof(float) * (size_t)planes * B * G) + Carver::round(sizeof(uint32_t) * (size_t)G * W) +
                6 * Carver::round(sizeof(int32_t) * (G + 4)) + Carver::round(sizeof(int64_t) * (G + 1)) +
                2 * Carver::round(sizeof(int32_t)) + (er ? Carver::round(sizeof(int32_t) * (size_t)B * er->P) : 0) +
                (edge_table ? Carver::round(sizeof(float) * (size_t)G * G) : 0) +
                3 * Carver::round(sizeof(int32_t) * rows) + 3 * Carver::round(sizeof(int4) * max_units) +
                Carver::round(sizeof(float2) * max_parts) + Carver::round(sizeof(float) * max_parts * ke) +
                Carver::round(sizeof(int32_t) * max_parts * ke) + Carver::round(sizeof(unsigned) * (size_t)B * kThrWords) +
                Carver::round(qg_bytes) + (smp ? Carver::round(sizeof(float) * (size_t)B * G) : 0) + (flat ? Carver::round(sizeof(int32_t) * rows) + Carver::round(sizeof(int32_t) * kg) : 0) + 8192;
  s = ensure_scratch(m, need);
  if (s != HTAM_OK) return s;
  Carver cv(m->scratch);
  float *s1 = cv.take<float>((size_t)planes * B * G);
  // The bitmap of the multi-kernel bucketing (group -> queries) lives in the
  // memory object and is zero between queries: the fill kernel clears each
  // word after its last read, so no memset precedes the bucketing.  A query
  // that stopped before the fill leaves it marked dirty; the next one clears
  // it first.
  uint32_t *bits = nullptr;
  int32_t *wpre = cv.take<int32_t>((size_t)G * W);
  int32_t *cnt = cv.take<int32_t>(G + 1);
  int32_t *bucket_off = cv.take<int32_t>(G + 1);
  int32_t *unit_off = cv.take<int32_t>(G + 1);
  int32_t *unit_off_tc = cv.take<int32_t>(G + 1);
  int32_t *unit_off_tc2 = cv.take<int32_t>(G + 1);
  int64_t *part_off = cv.take<int64_t>(G + 1);
  int32_t *n_units = cv.take<int32_t>(4);  // SIMT, single-SM and SM-pair tensor-core units
  int32_t *seg_tc = cv.take<int32_t>(1);        // pages per tensor-core unit, chosen on the device
  int32_t *tc_ctr = cv.take<int32_t>(2);        // tensor-core units taken from the shared counters
  int32_t *edge_prefix = er ? cv.take<int32_t>((size_t)B * er->P) : nullptr;
  float *edge_u = edge_table ? cv.take<float>((size_t)G * G) : nullptr;
  int32_t *bucket = cv.take<int32_t>(rows);
  int32_t *bucket_group = cv.take<int32_t>(rows);
  int32_t *pos = cv.take<int32_t>(rows);
  int4 *units = cv.take<int4>(max_units);
  int4 *units_tc = cv.take<int4>(max_units);
  int4 *units_tc2 = cv.take<int4>(max_units);
  float2 *part_ml = cv.take<float2>(max_parts);
  float *part_s = cv.take<float>(max_parts * ke);
  int32_t *part_id = cv.take<int32_t>(max_parts * ke);
  unsigned *thr_enc = cv.take<unsigned>((size_t)B * kThrWords);
  void *qg = q_gather ? static_cast<void *>(cv.take<char>(qg_bytes)) : nullptr;
  float *policy_keys = smp ? cv.take<float>((size_t)B * G) : nullptr;
  if (flat) {
    group_idx = cv.take<int32_t>(rows);
    int32_t *list = cv.take<int32_t>(kg);  // the non-empty groups, ascending
    mark.begin(HTAM_PHASE_SELECT);
    if (n_nonempty == 0) {
      HTAM_CK(cudaMemsetAsync(group_idx, 0xff, sizeof(int32_t) * (size_t)rows, st));
    } else {
      launch_kernel(flat_groups_kernel, 1, 1024, 0, st, m->count, G, list);
      HTAM_CK_LAUNCH("flat_groups_kernel");
      launch_kernel(flat_fill_kernel, (unsigned)ceil_div(rows, 256), 256, 0, st, list, rows, kg, group_idx);
      HTAM_CK_LAUNCH("flat_fill_kernel");
      mark.launched(2);
    }
    mark.end();
  }

  // 1. Coarse scores and the selected groups.
  if (!flat) {
    mark.begin(HTAM_PHASE_COARSE);
    if (er) {
      // Transition-edge scores (the prefix ids were checked on the host).
      HTAM_CK(cudaMemcpyAsync(edge_prefix, er->prefix, sizeof(int32_t) * (size_t)B * er->P,
                              cudaMemcpyHostToDevice, st));
      EdgeKernelArgs ea;
      ea.Z = er->Z;
      ea.prefix = edge_prefix;
      ea.F = er->F;
      ea.P = er->P;
      for (int f = 0; f < HTAM_MAX_EDGE_FEATURES; ++f) ea.w[f] = er->w[f];
      for (int i = 0; i < HTAM_MAX_PREFIX; ++i) ea.alpha[i] = er->alpha[i];
      if (edge_table) {
        launch_kernel(edge_phi_kernel, (unsigned)ceil_div((int64_t)G * G, 256), 256, 0, st, ea, G, edge_u);
        HTAM_CK_LAUNCH("edge_phi_kernel");
        launch_kernel(edge_gather_kernel, (unsigned)ceil_div((int64_t)B * G, 256), 256, 0, st, ea, edge_u, B, G, s1);
        HTAM_CK_LAUNCH("edge_gather_kernel");
        mark.launched();
      } else {
        launch_kernel(edge_scores_kernel, (unsigned)ceil_div((int64_t)B * G, 256), 256, 0, st, ea, B, G, s1);
        HTAM_CK_LAUNCH("edge_scores_kernel");
      }
    } else if (m->dtype == HTAM_BF16) {
      // Tensor cores against the split (hi + lo) bf16 group keys.
      s = launch_coarse_tc(queries, B, d, m->cent_hi, m->cent_lo, m->count, G, planes, s1, m->status, kMaxPolls,
                           st);
      if (s != HTAM_OK) return s;
    } else {
      // fp32 memories: CUDA cores against the fp32 keys.
      dim3 grid((unsigned)ceil_div(G, 64), (unsigned)ceil_div(B, 64));
      launch_kernel(coarse_scores_simt_kernel<float>, grid, 256, 0, st, static_cast<const float *>(queries), B, d,
                                                             m->cent, m->count, G, s1, nullptr);
      HTAM_CK_LAUNCH("coarse_scores_simt_kernel");
    }
    mark.launched();
    mark.end();
    mark.begin(HTAM_PHASE_SELECT);
    // Drawn groups (Algorithm 1, step 2): the top k_g of the policy keys.
    const float *sel = s1;
    int sel_planes = planes;
    if (smp) {
      if (n_nonempty > 0) {
        PolicyArgs pa{s1, planes, B, G, m->count, n_nonempty, 1.0f / p.tau, p.epsilon,
                      make_uint2((uint32_t)smp->seed, (uint32_t)(smp->seed >> 32)), (uint32_t)smp->offset,
                      (uint32_t)(smp->offset >> 32), policy_keys};
        launch_kernel(policy_keys_kernel, (unsigned)B, 256, 0, st, pa);
        HTAM_CK_LAUNCH("policy_keys_kernel");
        mark.launched();
      } else {
        HTAM_CK(cudaMemsetAsync(policy_keys, 0, sizeof(float) * (size_t)B * G, st));  // all groups empty
      }
      sel = policy_keys;
      sel_planes = 1;
    }
    const int swpq = select_warps_per_query(B, m->sm_count);
    if (swpq == 32) {
      launch_kernel(group_topk_kernel<32>, (unsigned)B, 32 * 32, 0, st, sel, sel_planes, B, G, m->count, kg, group_idx,
                                                            group_score, nullptr);
    } else if (swpq == 8) {
      launch_kernel(group_topk_kernel<8>, (unsigned)B, kSelWarps * 32, 0, st, sel, sel_planes, B, G, m->count, kg, group_idx,
                                                                   group_score, nullptr);
    } else if (swpq == 2) {
      launch_kernel(group_topk_kernel<2>, (unsigned)ceil_div(B, kSelWarps / 2), kSelWarps * 32, 0, st, sel, sel_planes, B,
                    G, m->count, kg, group_idx, group_score, nullptr);
    } else {
      launch_kernel(group_topk_kernel<1>, (unsigned)ceil_div(B, kSelWarps), kSelWarps * 32, 0, st,
          sel, sel_planes, B, G, m->count, kg, group_idx, group_score, nullptr);
    }
    HTAM_CK_LAUNCH("group_topk_kernel");
    mark.launched();
    if (smp) {
      launch_kernel(policy_scores_kernel, (unsigned)ceil_div((int64_t)B * kg, 256), 256, 0, st, s1, planes, B, G, kg,
                                                                                   group_idx, group_score);
      HTAM_CK_LAUNCH("policy_scores_kernel");
      mark.launched();
    }
    mark.end();
  }

  // 2. Buckets: group -> queries, work units, partial-record offsets.
  mark.begin(HTAM_PHASE_BUCKET);
  if ((int64_t)G * W <= kBucketSmallWords && rows <= kBucketSmallRows) {
    BucketSmallArgs ba{group_idx, B, kg, G, W, m->page_off, rt, m->sm_count, cnt, wpre, pos, bucket_off, unit_off,
                       unit_off_tc, unit_off_tc2, part_off, n_units, seg_tc, bucket, bucket_group, units, units_tc,
                       units_tc2, tc_ok ? thr_enc : nullptr, B * kThrWords, tc_ctr};
    static std::atomic<uint64_t> attr_set{0};
    if (first_on_device(attr_set)) {
      HTAM_CK(cudaFuncSetAttribute(bucket_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   (int)(sizeof(uint32_t) * kBucketSmallWords)));
    }
    launch_kernel(bucket_small_kernel, 1, 1024, sizeof(uint32_t) * (size_t)G * W, st, ba);
    HTAM_CK_LAUNCH("bucket_small_kernel");
    mark.launched();
  } else {
    if ((int64_t)G * W > m->qbits_len) {
      if (m->qbits) cudaFree(m->qbits);  // synchronises: no queued work still uses it
      m->qbits = nullptr;
      m->qbits_len = 0;
      const int64_t want = (int64_t)G * W + (int64_t)G * W / 2;
      if (cudaMalloc(&m->qbits, sizeof(uint32_t) * want) != cudaSuccess) {
        cudaGetLastError();
        m->qbits = nullptr;
        return HTAM_ENOMEM;
      }
      m->qbits_len = want;
      m->qbits_dirty = true;
    }
    bits = m->qbits;
    if (m->qbits_dirty) HTAM_CK(cudaMemsetAsync(bits, 0, sizeof(uint32_t) * (size_t)m->qbits_len, st));
    m->qbits_dirty = true;  // until the fill below is queued
    launch_kernel(bucket_bits_kernel, (unsigned)ceil_div(rows, 256), 256, 0, st, group_idx, B, kg, W, bits);
    HTAM_CK_LAUNCH("bucket_bits_kernel");
    launch_kernel(bucket_count_kernel, (unsigned)ceil_div((int64_t)G * 32, 256), 256, 0, st, bits, G, W, cnt, wpre);
    HTAM_CK_LAUNCH("bucket_count_kernel");
    launch_kernel(bucket_pos_kernel, (unsigned)ceil_div(rows, 256), 256, 0, st, bits, wpre, W, group_idx, rows, kg, pos);
    HTAM_CK_LAUNCH("bucket_pos_kernel");
    launch_kernel(bucket_scan_kernel, 1, 1024, 0, st, cnt, m->page_off, G, rt, m->sm_count, bucket_off, unit_off,
                                           unit_off_tc, unit_off_tc2, part_off, n_units, seg_tc);
    HTAM_CK_LAUNCH("bucket_scan_kernel");
    launch_kernel(bucket_fill_kernel, (unsigned)ceil_div((int64_t)G * 32, 256), 256, 0, st,
        bits, G, W, bucket_off, cnt, m->page_off, rt, seg_tc, unit_off, unit_off_tc, unit_off_tc2, bucket,
        bucket_group, units, units_tc, units_tc2, tc_ok ? thr_enc : nullptr, B * kThrWords, tc_ctr);
    HTAM_CK_LAUNCH("bucket_fill_kernel");
    m->qbits_dirty = false;
    mark.launched(5);
  }
  CUtensorMap q_map;
  if (tc_ok) {
    // Queries of tensor-core buckets in bucket order (the MMA's A operand),
    // and the per-query score bounds the tensor-core units share.
    if (!m->pool_map_ready) {
      s = make_bf16_tile_map(&m->pool_map, m->pool, (uint64_t)m->n_pages_max * kPageRows, d, kPageRows);
      if (s != HTAM_OK) return s;
      m->pool_map_ready = true;
    }
    // (A map of the query matrix when no bucket-ordered copy is made; the
    // kernel then ignores it unless the scan is flat.)
    s = q_gather ? make_bf16_tile_map(&q_map, qg, rows, d, kTcRows) : make_bf16_tile_map(&q_map, queries, B, d, kTcRows);
    if (s != HTAM_OK) return s;
    if (q_gather) {
      s = launch_gather_queries(queries, d, bucket, bucket_group, cnt, rt.tc_min, bucket_off + G, rows, qg, st);
      if (s != HTAM_OK) return s;
      mark.launched();
    }
  }
  mark.end();

  // 3a. Fine scores of small buckets on the CUDA cores.  When both fine
  // kernels run, the CUDA-core one goes to the memory's internal stream,
  // forked from the caller's stream here and joined back before the merge,
  // so that it shares the SMs with the tensor-core kernel instead of running
  // before it (the two write disjoint partial records).
  const bool overlap = tc_ok && m->fine_overlap;
  cudaStream_t fst = st;
  if (overlap) {
    if (!m->side) {
      if (cudaStreamCreateWithFlags(&m->side, cudaStreamNonBlocking) != cudaSuccess ||
          cudaEventCreateWithFlags(&m->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&m->ev_join, cudaEventDisableTiming) != cudaSuccess) {
        set_last_error("creating the internal stream", cudaGetLastError());
        return HTAM_ECUDA;
      }
    }
    HTAM_CK(cudaEventRecord(m->ev_fork, st));
    HTAM_CK(cudaStreamWaitEvent(m->side, m->ev_fork, 0));
    fst = m->side;
  }
  PhaseMark fmark(m, fst);
  fmark.begin(HTAM_PHASE_FINE);
  {
    // Rows prefetched into per-warp shared-memory rings; rows or query
    // blocks too large for the rings take direct 16-byte loads.
    StreamArgs sa{m->pool, d, m->slot_id, m->page_list, m->page_off, m->count, queries, bucket, bucket_off,
                  cnt, units, n_units, part_off, ke, 1.0f / p.tau, kSimtSegPages, part_ml, part_s, part_id};
    s = m->stream_rows ? launch_fine_stream(sa, qc, m->dtype, m->sm_count, fst) : HTAM_EINVAL;
    if (s == HTAM_EINVAL) {
      FineArgs fa{m->pool, d, m->slot_id, m->page_list, m->page_off, m->count, queries, bucket, bucket_off,
                  cnt, units, n_units, part_off, ke, 1.0f / p.tau, kSimtSegPages, part_ml, part_s, part_id};
      s = m->dtype == HTAM_BF16 ? dispatch_fine_simt<__nv_bfloat16>(qc, fa, m->sm_count, max_units, fst)
                                : dispatch_fine_simt<float>(qc, fa, m->sm_count, max_units, fst);
    }
  }
  if (s != HTAM_OK) return s;
  fmark.launched();
  fmark.end();
  if (overlap) HTAM_CK(cudaEventRecord(m->ev_join, fst));

  // 3b. Fine scores of large buckets on the tensor cores.
  if (tc_ok) {
    mark.begin(HTAM_PHASE_FINE_TC);
    TcFineArgs ta{units_tc, n_units + 1, tc_ctr, bucket, bucket_off, cnt, m->page_list, m->page_off, m->count, m->slot_id,
                  part_off, d, seg_tc, ke, 1.4426950408889634f / p.tau, part_ml, part_s, part_id, thr_enc,
                  m->status, kMaxPolls, flat ? 1 : 0, a_rows ? 1 : 0,
                  static_cast<const uint4 *>(queries), d * 2 / 16};
    if (tc_pairs_run) {
      // Buckets of several chunks on SM pairs, then the one-chunk buckets
      // (both by TMA: from the bucket-ordered copy, or the query matrix in a
      // flat scan).
      TcFineArgs tp = ta;
      tp.units = units_tc2;
      tp.n_units = n_units + 2;
      tp.unit_ctr = tc_ctr + 1;
      s = launch_fine_tc(tp, q_map, m->pool_map, 2 * (int)std::min<int64_t>(max_units, m->sm_count / 2), true, st);
      if (s != HTAM_OK) return s;
      mark.launched();
    }
    s = launch_fine_tc(ta, q_map, m->pool_map, (int)std::min<int64_t>(max_units, m->sm_count), false, st);
    if (s != HTAM_OK) return s;
    mark.launched();
    mark.end();
  }

  if (overlap) HTAM_CK(cudaStreamWaitEvent(st, m->ev_join, 0));

  // 4. Merge per query.
  mark.begin(HTAM_PHASE_MERGE);
  MergeArgs ma{group_idx, B, kg, ke, m->count, pos, cnt, m->page_off, rt, seg_tc, part_off, part_ml, part_s,
               part_id, 1.0f / p.tau, p.epsilon, entry_idx, entry_score, entry_weight, lse};
  if (wpq == 8) {
    launch_kernel(merge_kernel<8>, (unsigned)B, kMergeWarps * 32, 0, st, ma);
  } else {
    launch_kernel(merge_kernel<1>, (unsigned)ceil_div(B, kMergeWarps), kMergeWarps * 32, 0, st, ma);
  }
  HTAM_CK_LAUNCH("merge_kernel");
  mark.launched();
  mark.end();
  return HTAM_OK;
}

// ------------------------------------------------- nearest-key assignment

namespace {

// ids[i] = gid[i] when given, else the nearest group picked for row i.  gid
// and ids may be the same array (each thread reads and writes only its row).
// Rows appended without a group (id -1): the group picked for each, counted
// into the batch's group sizes; a row with no non-empty group to join marks
// the batch bad.  Gated on the batch's count of such rows.
__global__ void assign_resolve_kernel(const int32_t *__restrict__ gid, const int32_t *__restrict__ pick, int64_t n,
                                      const int32_t *__restrict__ gate, int32_t *__restrict__ ids,
                                      int32_t *__restrict__ bcount, int32_t *__restrict__ bad,
                                      int32_t *__restrict__ hist, int64_t row0, int64_t chunk, int64_t n_chunks) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  if (*gate == 0) return;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < n; t += (int64_t)gridDim.x * blockDim.x) {
    if (gid[t] != -1) continue;
    const int32_t p = pick[t];
    if (p < 0) {
      atomicOr(bad, 1);
    } else {
      ids[t] = p;
      atomicAdd(&bcount[p], 1);
      atomicAdd(&hist[(int64_t)p * n_chunks + (row0 + t) / chunk], 1);
    }
  }
}

}  // namespace

htam_status assign_unassigned(htam_memory *m, const void *entries, const int32_t *gid, int64_t count,
                              const int32_t *n_unassigned, int32_t *ids, int32_t *bcount, int32_t *bad,
                              int32_t *hist, int64_t chunk, int64_t n_chunks, cudaStream_t st, PhaseMark *mark) {
  const int G = m->n_groups, d = m->d;
  // Rows per pass: the [rows, G] score matrix stays within 16 MiB per plane.
  const int64_t R = std::max<int64_t>(1, std::min<int64_t>(count, (int64_t(1) << 22) / G));
  const int64_t last = count - (ceil_div(count, R) - 1) * R;
  auto planes_of = [&](int64_t rb) {
    return m->dtype == HTAM_BF16 ? coarse_tc_splits((int)rb, d, G, m->sm_count) : 1;
  };
  const int64_t s1_elems = std::max<int64_t>(planes_of(R) * R, planes_of(last) * last) * G;
  const size_t need = Carver::round(sizeof(float) * s1_elems) + Carver::round(sizeof(int32_t) * R) +
                      Carver::round(sizeof(float) * R) + 1024;
  if (need > m->assign_bytes) {
    if (m->assign_buf) cudaFree(m->assign_buf);  // synchronises: no queued work still reads it
    m->assign_buf = nullptr;
    m->assign_bytes = 0;
    const size_t want = need + need / 2;
    if (cudaMalloc(&m->assign_buf, want) != cudaSuccess) {
      cudaGetLastError();
      return HTAM_ENOMEM;
    }
    m->assign_bytes = want;
  }
  Carver cv(m->assign_buf);
  float *s1 = cv.take<float>(s1_elems);
  int32_t *pick = cv.take<int32_t>(R);
  float *pick_score = cv.take<float>(R);
  for (int64_t r0 = 0; r0 < count; r0 += R) {
    const int rb = (int)std::min<int64_t>(R, count - r0);
    const void *rows = static_cast<const char *>(entries) + r0 * d * m->elem_bytes;
    const int planes = planes_of(rb);
    if (m->dtype == HTAM_BF16) {
      htam_status s = launch_coarse_tc(rows, rb, d, m->cent_hi, m->cent_lo, m->count, G, planes, s1, m->status,
                                       kMaxPolls, st, n_unassigned);
      if (s != HTAM_OK) return s;
    } else {
      dim3 grid((unsigned)ceil_div(G, 64), (unsigned)ceil_div(rb, 64));
      launch_kernel(coarse_scores_simt_kernel<float>, grid, 256, 0, st, static_cast<const float *>(rows), rb, d, m->cent,
                                                             m->count, G, s1, n_unassigned);
      HTAM_CK_LAUNCH("coarse_scores_simt_kernel");
    }
    if (warps_per_query(rb, m->sm_count) == 8) {
      launch_kernel(group_topk_kernel<8>, (unsigned)rb, kSelWarps * 32, 0, st, s1, planes, rb, G, m->count, 1, pick,
                                                                    pick_score, n_unassigned);
    } else {
      launch_kernel(group_topk_kernel<1>, (unsigned)ceil_div(rb, kSelWarps), kSelWarps * 32, 0, st,
          s1, planes, rb, G, m->count, 1, pick, pick_score, n_unassigned);
    }
    HTAM_CK_LAUNCH("group_topk_kernel");
    const unsigned blocks = (unsigned)std::min<int64_t>(ceil_div(rb, 256), 1024);
    launch_kernel(assign_resolve_kernel, blocks, 256, 0, st, gid + r0, pick, rb, n_unassigned, ids + r0, bcount, bad, hist, r0, chunk,
                  n_chunks);
    HTAM_CK_LAUNCH("assign_resolve_kernel");
    if (mark) mark->launched(3);
  }
  return HTAM_OK;
}

}  // namespace htam
