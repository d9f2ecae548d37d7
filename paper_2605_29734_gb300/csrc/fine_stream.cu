// fine_stream.cu -- fine scores of small buckets on the CUDA cores, with the
// selected groups' entry rows streamed through a shared-memory ring.
//
// Work unit = (group g, bucket chunk c, page segment s): up to QC queries
// that selected g (the Eq. 12 restriction) against the rows of a few pages of
// g.  The rows are read from HBM exactly once per unit by one producer thread
// issuing bulk asynchronous copies (cp.async.bulk, completion counted on an
// mbarrier) into a ring of 20 stages of up to 8 KiB (160 KiB in flight per
// SM, independent of registers); eight consumer warps take the stages
// round-robin, and the copies of later stages -- including those of the
// CTA's next unit -- are in flight while earlier ones are being scored.
//
// A consumer warp scores one row at a time: each lane reads 16-byte slices of
// the row and of the queries (kept in shared memory in the rows' own layout,
// so both reads are conflict-free), accumulates four independent partial dot
// products per query, and the warp reduces them with shuffles.  Per query the
// warp keeps the online softmax statistics of s/tau (the Eq. 11 normaliser)
// and a warp-distributed sorted top-k (the Eq. 13 pick as a top-k).  At the
// end of a unit the eight warps' states are merged per query and one partial
// record per (query, unit) is written for the merge kernel.  Every mbarrier
// wait is bounded.

#include <algorithm>

#include "common.cuh"
#include "fine_stream.h"
#include "sm100.cuh"

namespace htam {

namespace {

using namespace sm100;

constexpr int kConsumers = 8;                     // consumer warps
constexpr int kThreadsS = (kConsumers + 1) * 32;  // + one producer warp
constexpr int kRing = 20;                         // stages
constexpr int kStageBytes = kStreamMaxRowBytes;   // 8 KiB

template <typename T>
struct Vec16;
template <>
struct Vec16<__nv_bfloat16> {
  static constexpr int kN = 8;
  __device__ static void run(const uint4 &w, float *f) {
    f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
    f[4] = bf16lo(w.z); f[5] = bf16hi(w.z); f[6] = bf16lo(w.w); f[7] = bf16hi(w.w);
  }
};
template <>
struct Vec16<float> {
  static constexpr int kN = 4;
  __device__ static void run(const uint4 &w, float *f) {
    f[0] = __uint_as_float(w.x); f[1] = __uint_as_float(w.y);
    f[2] = __uint_as_float(w.z); f[3] = __uint_as_float(w.w);
  }
};

struct __align__(8) StreamBars {
  uint64_t full[kRing];
  uint64_t empty[kRing];
  int abort;
};

// Rows per stage: a power of two dividing the 128-row page, at most 32.
__host__ __device__ inline int rows_per_stage(int row_bytes) {
  int r = 1;
  while (r < 32 && (r * 2) * row_bytes <= kStageBytes) r *= 2;
  return r;
}

__host__ __device__ inline size_t stream_smem_bytes(int qc, int row_bytes) {
  return (size_t)kRing * kStageBytes + (size_t)qc * row_bytes +
         (sizeof(float) + sizeof(int)) * kConsumers * qc * 64 + sizeof(float) * 2 * kConsumers * qc +
         sizeof(StreamBars);
}

// acc += <16 bytes of row, 16 bytes of query>, element by element.
template <typename T>
__device__ __forceinline__ float dot16(const uint4 &row, const uint4 &q, float acc) {
  float f[Vec16<T>::kN], g[Vec16<T>::kN];
  Vec16<T>::run(row, f);
  Vec16<T>::run(q, g);
#pragma unroll
  for (int t = 0; t < Vec16<T>::kN; ++t) acc = fmaf(f[t], g[t], acc);
  return acc;
}

template <typename T, int QC>
__global__ void __launch_bounds__(kThreadsS, 1) fine_stream_kernel(StreamArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int d = a.d;
  const int row_bytes = d * (int)sizeof(T);
  const int n_vec = row_bytes / 16;
  const int R = rows_per_stage(row_bytes);
  uint8_t *ring = smem_raw;                                           // [kRing][kStageBytes]
  uint4 *qv = reinterpret_cast<uint4 *>(ring + kRing * kStageBytes);  // [QC][n_vec], rows' layout
  float *ws = reinterpret_cast<float *>(qv + QC * n_vec);             // [warps][QC][64]
  int *wi = reinterpret_cast<int *>(ws + kConsumers * QC * 64);       // [warps][QC][64]
  float *wm = reinterpret_cast<float *>(wi + kConsumers * QC * 64);   // [warps][QC]
  float *wl = wm + kConsumers * QC;                                   // [warps][QC]
  StreamBars *bars = reinterpret_cast<StreamBars *>(wl + kConsumers * QC);
  volatile int *abort = &bars->abort;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    for (int s = 0; s < kRing; ++s) {
      mbar_init(&bars->full[s], 1);
      mbar_init(&bars->empty[s], 1);
    }
    bars->abort = 0;
    fence_barrier_init();
  }
  __syncthreads();
  const int n_units = *a.n_units;
  const uint8_t *pool = static_cast<const uint8_t *>(a.pool);

  if (warp == kConsumers) {
    // ----------------------------------------------------------- producer
    uint32_t t = 0;  // stage batches issued by this CTA
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      const int4 U = a.units[u];
      const int g = U.x;
      const int pg0 = a.page_off[g];
      const int npg = a.page_off[g + 1] - pg0;
      const int p_beg = U.z * a.seg_pages, p_end = min(npg, p_beg + a.seg_pages);
      const int cnt_rows = a.count[g];
      for (int p = p_beg; ok && p < p_end; ++p) {
        const int fill = min(kPageRows, cnt_rows - p * kPageRows);
        const int64_t page_row = (int64_t)a.page_list[pg0 + p] * kPageRows;
        for (int r0 = 0; r0 < fill; r0 += R, ++t) {
          const int slot = t % kRing;
          if (!mbar_wait(&bars->empty[slot], ((t / kRing) & 1u) ^ 1u, abort, a.max_polls)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            const uint32_t bytes = (uint32_t)(min(R, fill - r0) * row_bytes);
            mbar_arrive_expect_tx(&bars->full[slot], bytes);
            bulk_load(smem_addr(ring + slot * kStageBytes), pool + (page_row + r0) * row_bytes, bytes,
                      &bars->full[slot]);
          }
          __syncwarp();
        }
      }
    }
    if (!ok && lane == 0) {
      atomicOr(a.status, 1u);
      bars->abort = 1;
    }
    // Drain: the copies of the last kRing batches have landed.
    for (uint32_t back = 1; back <= kRing && back <= t; ++back) {
      const uint32_t tt = t - back;
      for (uint32_t i = 0; i < a.max_polls && !mbar_try_wait(&bars->full[tt % kRing], (tt / kRing) & 1u); ++i) {
      }
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------- consumers
    // After a give-up (ok == false) a warp keeps walking the same units and
    // batches -- its waits then return at once -- so that every consumer
    // warp reaches every named barrier.
    const T *Q = static_cast<const T *>(a.Q);
    const int ke = a.ke;
    uint32_t t = 0;  // stage batches seen by this CTA (all consumer warps count them all)
    bool ok = true;
    for (int u = blockIdx.x; u < n_units; u += gridDim.x) {
      const int4 U = a.units[u];
      const int g = U.x, c = U.y, s = U.z;
      const int cg = a.cnt[g];
      const int q0 = c * QC;
      const int nq = min(QC, cg - q0);
      const int *bq = a.bucket + a.bucket_off[g] + q0;

      // Stage the unit's queries in the rows' layout (the previous unit is
      // done with them).
      for (int i = tid; i < nq * n_vec; i += kConsumers * 32) {
        const int j = i / n_vec, v = i % n_vec;
        qv[j * n_vec + v] = reinterpret_cast<const uint4 *>(Q + (int64_t)bq[j] * d)[v];
      }
      named_sync(1, kConsumers * 32);

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

      const int pg0 = a.page_off[g];
      const int npg = a.page_off[g + 1] - pg0;
      const int p_beg = s * a.seg_pages, p_end = min(npg, p_beg + a.seg_pages);
      const int cnt_rows = a.count[g];
      for (int p = p_beg; p < p_end; ++p) {
        const int fill = min(kPageRows, cnt_rows - p * kPageRows);
        const int64_t page_row = (int64_t)a.page_list[pg0 + p] * kPageRows;
        for (int r0 = 0; r0 < fill; r0 += R, ++t) {
          if ((int)(t % kConsumers) != warp) continue;
          const int slot = t % kRing;
          const int nrows = min(R, fill - r0);
          const int my_id = lane < nrows ? a.slot_id[page_row + r0 + lane] : INT_MAX;
          if (ok && !mbar_wait(&bars->full[slot], (t / kRing) & 1u, abort, a.max_polls)) ok = false;
          if (!ok) continue;
          const uint4 *stage = reinterpret_cast<const uint4 *>(ring + slot * kStageBytes);
          for (int rr = 0; rr < nrows; ++rr) {
            const uint4 *row = stage + rr * n_vec;
            const int id = __shfl_sync(kFullMask, my_id, rr);
            // Four independent partial sums per query (vectors v, v+32, v+64,
            // v+96 of each group of 128) keep the FMA pipeline busy.
            float acc[QC][4];
#pragma unroll
            for (int j = 0; j < QC; ++j)
#pragma unroll
              for (int k = 0; k < 4; ++k) acc[j][k] = 0.f;
            for (int v0 = lane; v0 < n_vec; v0 += 128) {
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int v = v0 + 32 * k;
                if (v < n_vec) {
                  const uint4 w = row[v];
#pragma unroll
                  for (int j = 0; j < QC; ++j) {
                    if (j < nq) acc[j][k] = dot16<T>(w, qv[j * n_vec + v], acc[j][k]);
                  }
                }
              }
            }
#pragma unroll
            for (int j = 0; j < QC; ++j) {
              if (j < nq) {
                const float sc = warp_sum((acc[j][0] + acc[j][1]) + (acc[j][2] + acc[j][3]));
                const float z = sc * a.inv_tau;
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
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->empty[slot]);
        }
      }

      // Merge the eight warps' states per query and write the partial records.
#pragma unroll
      for (int j = 0; j < QC; ++j) {
        if (j < nq) {
          const int o = (warp * QC + j) * 64;
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
      named_sync(1, kConsumers * 32);
      for (int j = warp; ok && j < nq; j += kConsumers) {
        float M = -INFINITY;
        for (int w = 0; w < kConsumers; ++w) M = fmaxf(M, wm[w * QC + j]);
        float Ls = 0.f;
        for (int w = 0; w < kConsumers; ++w) {
          const float mw = wm[w * QC + j];
          if (mw != -INFINITY) Ls += wl[w * QC + j] * expf(mw - M);
        }
        WarpList F;
        F.init();
        float fs = -INFINITY;
        int fi = INT_MAX;
        for (int w = 0; w < kConsumers; ++w) {
          for (int h = 0; h < 2; ++h) {
            if (h * 32 >= ke) break;
            const int o = (w * QC + j) * 64 + h * 32;
            const float cs = ws[o + lane];
            const int ci = wi[o + lane];
            unsigned mask = __ballot_sync(kFullMask, h * 32 + lane < ke && ci != INT_MAX && better(cs, ci, fs, fi));
            while (mask) {
              const int src = __ffs(mask) - 1;
              mask &= mask - 1;
              const float vs = __shfl_sync(kFullMask, cs, src);
              const int vi = __shfl_sync(kFullMask, ci, src);
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
      named_sync(1, kConsumers * 32);  // shared state is free for the next unit
    }
    if (!ok && lane == 0) {
      atomicOr(a.status, 1u);
      bars->abort = 1;
    }
  }
  __syncthreads();
}

template <typename T, int QC>
htam_status launch_qc(const StreamArgs &a, int sm_count, cudaStream_t st) {
  const size_t smem = stream_smem_bytes(QC, a.d * (int)sizeof(T));
  if (smem > 227 * 1024) return HTAM_EINVAL;
  auto kernel = fine_stream_kernel<T, QC>;
  HTAM_CK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  kernel<<<sm_count, kThreadsS, smem, st>>>(a);
  HTAM_CK_LAUNCH("fine_stream_kernel");
  return HTAM_OK;
}

template <typename T>
htam_status launch_t(const StreamArgs &a, int qc, int sm_count, cudaStream_t st) {
  switch (qc) {
    case 8: return launch_qc<T, 8>(a, sm_count, st);
    case 4: return launch_qc<T, 4>(a, sm_count, st);
    case 2: return launch_qc<T, 2>(a, sm_count, st);
    default: return launch_qc<T, 1>(a, sm_count, st);
  }
}

}  // namespace

htam_status launch_fine_stream(const StreamArgs &a, int qc, htam_dtype dtype, int sm_count, cudaStream_t st) {
  const int row_bytes = a.d * (dtype == HTAM_BF16 ? 2 : 4);
  if (row_bytes > kStreamMaxRowBytes || row_bytes % 16 != 0) return HTAM_EINVAL;
  // With one row per stage each consumer warp has too little prefetched
  // (measured slower than direct loads on 8 KiB rows): stream only when a
  // stage holds at least two rows.
  if (rows_per_stage(row_bytes) < 2) return HTAM_EINVAL;
  return dtype == HTAM_BF16 ? launch_t<__nv_bfloat16>(a, qc, sm_count, st) : launch_t<float>(a, qc, sm_count, st);
}

}  // namespace htam
