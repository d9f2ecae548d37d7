// fine_stream.cu -- fine scores of small buckets on the CUDA cores (bf16
// memories), with the selected groups' entry rows prefetched into per-warp
// shared-memory rings.
//
// Work unit = (group g, bucket chunk c, page segment s): up to QC queries
// that selected g (the Eq. 12 restriction) against the rows of a few pages of
// g, each row read from HBM once per unit.  Warp w of the block scores rows
// w, w+8, ... of the unit.
//
// Rows: every lane copies its own 16-byte slices of the warp's upcoming rows
// into the warp's ring with cp.async (L1 bypassed) a few rows ahead of the
// row it is scoring, then reads back exactly those slices: no lane waits for
// another lane's copy, no barrier guards a ring slot, and the bytes in flight
// sit in shared memory, not in registers.  Lane 0 copies each row's entry id
// along with the row.  The ring depth is a compile-time function of the
// query block and of the longest row the instantiation serves, so the waits
// and slot indices are constants.  The copies of a unit's first rows are
// issued before the previous unit's warps are merged, so the row stream
// does not pause between units.
//
// Queries: the registers left free by the ring hold each lane's slices of
// the unit's queries as packed bf16 (QC x KV x 16 bytes), so scoring a row
// reads shared memory once per row slice; the products go through the
// mixed-precision fma.rn.f32.bf16 (bf16 operands, fp32 accumulator).  A
// product of two bf16 values is exact in fp32, so this rounds exactly like
// widening both operands and calling fmaf.  The partial sums of a query (one
// per slice of the lane, or two for 8-query blocks) are reduced across the warp with shuffles; per query the warp keeps the online
// softmax statistics of s/tau (the Eq. 11 normaliser) and a warp-distributed
// sorted top-k (the Eq. 13 pick as a top-k, k_entries <= 32), both updated
// 32 rows at a time.  At the end of a unit the eight
// warps' states are merged per query and one partial record per (query,
// unit) is written for the merge kernel.

#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "fine_stream.h"

namespace htam {

namespace {

constexpr int kWarps = 8;
constexpr int kMaxSlots = 16;           // rows per warp ring: cp.async.wait_group takes at most 15 pending
constexpr int kMaxSegPages = 4;         // pages of a unit, held in registers
constexpr int kSmemLimit = 227 * 1024;  // opt-in dynamic shared memory per block
constexpr int kMaxQueryVecs = 32;       // QC x KV: 128 registers of packed queries

// Shared memory besides the row rings: row ids, per-warp top-k lists (32
// slots: k_entries <= 32) and softmax statistics.
__host__ __device__ constexpr size_t side_bytes(int qc) {
  return sizeof(int) * kWarps * kMaxSlots + (sizeof(float) + sizeof(int)) * kWarps * qc * 32 +
         sizeof(float) * 2 * kWarps * qc;
}

// Ring depth (rows per warp) for QC queries per unit and rows of up to
// 32 * KV 16-byte slices: as many as the shared memory holds, at most 16.
template <int QC, int KV>
__host__ __device__ constexpr int ring_slots() {
  const size_t per_slot = (size_t)kWarps * KV * 32 * 16;
  const size_t n = (kSmemLimit - side_bytes(QC)) / per_slot;
  return n < (size_t)kMaxSlots ? (int)n : kMaxSlots;
}

__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async4(void *smem_dst, const void *gmem_src) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// acc + x.lo * y.lo + x.hi * y.hi for two packed bf16 pairs, fp32 accumulate.
__device__ __forceinline__ float fma_bf16x2(uint32_t x, uint32_t y, float acc) {
  asm("{\n\t.reg .b16 xl, xh, yl, yh;\n\t"
      "mov.b32 {xl, xh}, %1;\n\t"
      "mov.b32 {yl, yh}, %2;\n\t"
      "fma.rn.f32.bf16 %0, xl, yl, %0;\n\t"
      "fma.rn.f32.bf16 %0, xh, yh, %0;\n\t}"
      : "+f"(acc)
      : "r"(x), "r"(y));
  return acc;
}

// acc + <8 bf16 of a row, 8 bf16 of a query>, in element order.
__device__ __forceinline__ float dot8_bf16(const uint4 &w, const uint4 &q, float acc) {
  acc = fma_bf16x2(w.x, q.x, acc);
  acc = fma_bf16x2(w.y, q.y, acc);
  acc = fma_bf16x2(w.z, q.z, acc);
  return fma_bf16x2(w.w, q.w, acc);
}

// Where one warp's rows of one unit are.
struct UnitRows {
  int g, q0, nq, cg, s, r0, my_rows;
  int pg[kMaxSegPages];  // storage pages of the unit's segment
};

template <int QC>
__device__ __forceinline__ UnitRows unit_rows(const StreamArgs &a, int u, int warp) {
  const int4 U = a.units[u];
  UnitRows r;
  r.g = U.x;
  r.s = U.z;
  r.cg = a.cnt[r.g];
  r.q0 = U.y * QC;
  r.nq = min(QC, r.cg - r.q0);
  const int pg0 = a.page_off[r.g];
  const int npages = a.page_off[r.g + 1] - pg0;
  const int p_beg = r.s * a.seg_pages;
  const int p_end = min(npages, p_beg + a.seg_pages);
#pragma unroll
  for (int k = 0; k < kMaxSegPages; ++k) r.pg[k] = p_beg + k < p_end ? a.page_list[pg0 + p_beg + k] : 0;
  r.r0 = p_beg * kPageRows;
  const int r1 = min(p_end * kPageRows, a.count[r.g]);
  r.my_rows = r1 - r.r0 > warp ? (r1 - r.r0 - warp + kWarps - 1) / kWarps : 0;
  return r;
}

template <int QC, int KV>
__global__ void __launch_bounds__(kWarps * 32, 1) fine_ring_kernel(StreamArgs a) {
  pdl_entry();  // after the previous kernel of the stream (see common.cuh)
  // Slice t of a lane is row slice lane + 32 t, and query register qr[j][t]
  // holds the same slice of query j.
  constexpr int S = ring_slots<QC, KV>();
  constexpr int AHEAD = S - 1;  // rows in flight beyond the one being scored
  // Partial sums per query: one per slice, two when eight queries already
  // fill the registers.
  constexpr int NP = QC >= 8 && KV > 2 ? 2 : KV;
  // Ring slots are 32 * KV slices long whatever the row length; the slices
  // past the row stay zero, so scoring needs no bounds test.
  constexpr int RS = 32 * KV;
  static_assert(S >= kStreamMinSlots, "ring too shallow");
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int n_vec = a.d / 8;  // 16-byte slices per row, at most RS
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint4 *ring = reinterpret_cast<uint4 *>(smem_raw) + (size_t)warp * S * RS;  // this warp's ring
  int *ids_all = reinterpret_cast<int *>(reinterpret_cast<uint4 *>(smem_raw) + (size_t)kWarps * S * RS);
  int *ids = ids_all + warp * kMaxSlots;                             // this warp's row ids
  float *ws = reinterpret_cast<float *>(ids_all + kWarps * kMaxSlots);  // [warps][QC][32]
  int *wi = reinterpret_cast<int *>(ws + kWarps * QC * 32);            // [warps][QC][32]
  float *wm = reinterpret_cast<float *>(wi + kWarps * QC * 32);        // [warps][QC]
  float *wl = wm + kWarps * QC;                                        // [warps][QC]
  const int n_units = *a.n_units;
  const uint4 *pool = static_cast<const uint4 *>(a.pool);
  const uint4 *Q = static_cast<const uint4 *>(a.Q);
  const int ke = a.ke;

  // Copies this lane's slices of row i of unit U, and on lane 0 the row's
  // entry id, into ring slot i % S.  One copy group per row, empty past the
  // unit's last row, keeps the count of groups equal to the count of rows.
  auto prefetch = [&](const UnitRows &U, int i) {
    if (i < U.my_rows) {
      const int r = U.r0 + warp + i * kWarps;  // row of the group; r0 is page-aligned
      const int pi = (r - U.r0) / kPageRows;
      const int page = pi == 0 ? U.pg[0] : pi == 1 ? U.pg[1] : pi == 2 ? U.pg[2] : U.pg[3];
      const int64_t slot = (int64_t)page * kPageRows + (r % kPageRows);
      const int k = i % S;
      const uint4 *src = pool + slot * n_vec;
      uint4 *dst = ring + k * RS;
#pragma unroll
      for (int t = 0; t < KV; ++t) {
        const int o = lane + 32 * t;
        if (o < n_vec) cp_async16(dst + o, src + o);
      }
      if (lane == 0) cp_async4(ids + k, a.slot_id + slot);
    }
    cp_async_commit();
  };

  // Zero the slices past the row once; copies never write them, and each is
  // read only by the lane that zeroed it.
  if (n_vec < RS) {
#pragma unroll
    for (int k = 0; k < S; ++k)
#pragma unroll
      for (int t = 0; t < KV; ++t) {
        const int o = lane + 32 * t;
        if (o >= n_vec) ring[k * RS + o] = make_uint4(0u, 0u, 0u, 0u);
      }
  }

  int u = blockIdx.x;
  UnitRows cur{};
  if (u < n_units) {
    cur = unit_rows<QC>(a, u, warp);
#pragma unroll
    for (int i = 0; i < AHEAD; ++i) prefetch(cur, i);
  }
  for (; u < n_units; u += gridDim.x) {
    const int nq = cur.nq;
    uint4 qr[QC][KV];
    {
      const int *bq = a.bucket + a.bucket_off[cur.g] + cur.q0;
#pragma unroll
      for (int j = 0; j < QC; ++j) {
        const int64_t qrow = j < nq ? (int64_t)bq[j] * n_vec : 0;
#pragma unroll
        for (int t = 0; t < KV; ++t) {
          const int o = lane + 32 * t;
          qr[j][t] = j < nq && o < n_vec ? Q[qrow + o] : make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }

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
    // The row loop with the unit's query count NQ as a constant, so the
    // slices of a row feed NQ x KV independent FMA chains in one block.  Row
    // scores are buffered one row per lane and taken in 32 rows at a time:
    // one warp max and one warp sum update the softmax statistics, and only
    // if some buffered row can enter the top-k (k_entries <= 32) are the 32
    // sorted across the warp and merged into the list.
    auto score_rows = [&](auto nq_c) {
      constexpr int NQ = decltype(nq_c)::value;
      float bs[NQ];  // lane r: the score of buffered row r
      int bid = INT_MAX;
      auto flush = [&](int nv) {
        const bool in = lane < nv;
#pragma unroll
        for (int j = 0; j < NQ; ++j) {
          const float z = in ? bs[j] * a.inv_tau : -INFINITY;
          const float zm = warp_max(z);
          if (zm > m[j]) {
            l[j] *= expf(m[j] - zm);
            m[j] = zm;
          }
          l[j] += warp_sum(in ? expf(z - m[j]) : 0.f);
          float cs = in ? bs[j] : -INFINITY;
          int ci = in ? bid : INT_MAX;
          if (__any_sync(kFullMask, in && better(cs, ci, ts[j], ti[j]))) {
            warp_sort32(cs, ci);
            lst[j].merge32(cs, ci);
            lst[j].kth(ke, ts[j], ti[j]);
          }
        }
      };
      for (int i = 0; i < cur.my_rows; ++i) {
        prefetch(cur, i + AHEAD);
        cp_async_wait<AHEAD>();  // row i has landed; rows i+1 .. i+AHEAD may still be pending
        const int ks = i % S;
        const uint4 *row = ring + ks * RS;
        const int id = __shfl_sync(kFullMask, lane == 0 ? ids[ks] : 0, 0);
        float acc[NQ][NP];
#pragma unroll
        for (int j = 0; j < NQ; ++j)
#pragma unroll
          for (int t = 0; t < NP; ++t) acc[j][t] = 0.f;
#pragma unroll
        for (int t = 0; t < KV; ++t) {
          const uint4 w = row[lane + 32 * t];
#pragma unroll
          for (int j = 0; j < NQ; ++j) acc[j][t % NP] = dot8_bf16(w, qr[j][t], acc[j][t % NP]);
        }
        const bool mine = lane == (i & 31);
#pragma unroll
        for (int j = 0; j < NQ; ++j) {
#pragma unroll
          for (int h = NP / 2; h >= 1; h /= 2)
#pragma unroll
            for (int t = 0; t < h; ++t) acc[j][t] += acc[j][t + h];
          const float sc = warp_sum(acc[j][0]);
          if (mine) bs[j] = sc;
        }
        if (mine) bid = id;
        if ((i & 31) == 31 || i + 1 == cur.my_rows) flush((i & 31) + 1);
      }
    };
    switch (nq) {
      case 1: score_rows(std::integral_constant<int, 1>{}); break;
      case 2: if constexpr (QC >= 2) score_rows(std::integral_constant<int, 2>{}); break;
      case 3: if constexpr (QC >= 4) score_rows(std::integral_constant<int, 3>{}); break;
      case 4: if constexpr (QC >= 4) score_rows(std::integral_constant<int, 4>{}); break;
      case 5: if constexpr (QC >= 8) score_rows(std::integral_constant<int, 5>{}); break;
      case 6: if constexpr (QC >= 8) score_rows(std::integral_constant<int, 6>{}); break;
      case 7: if constexpr (QC >= 8) score_rows(std::integral_constant<int, 7>{}); break;
      case 8: if constexpr (QC >= 8) score_rows(std::integral_constant<int, 8>{}); break;
    }

    // Every copy still pending belongs to an empty group, and this lane has
    // read all of its slices: start the next unit's rows now.
    const UnitRows done = cur;
    if (u + (int)gridDim.x < n_units) {
      cur = unit_rows<QC>(a, u + gridDim.x, warp);
#pragma unroll
      for (int i = 0; i < AHEAD; ++i) prefetch(cur, i);
    }

    // Hand each warp's state to shared memory, then warp j merges query j.
    __syncthreads();  // the previous unit's merge is done reading
#pragma unroll
    for (int j = 0; j < QC; ++j) {
      if (j < nq) {
        const int o = (warp * QC + j) * 32;
        ws[o + lane] = lst[j].s0;
        wi[o + lane] = lst[j].i0;
        if (lane == 0) {
          wm[warp * QC + j] = m[j];
          wl[warp * QC + j] = l[j];
        }
      }
    }
    __syncthreads();
    for (int j = warp; j < nq; j += kWarps) {
      float M = -INFINITY;
      for (int w = 0; w < kWarps; ++w) M = fmaxf(M, wm[w * QC + j]);
      float Ls = 0.f;
      for (int w = 0; w < kWarps; ++w) {
        const float mw = wm[w * QC + j];
        if (mw != -INFINITY) Ls += wl[w * QC + j] * expf(mw - M);
      }
      WarpList F;
      F.init();
      float fs = -INFINITY;
      int fi = INT_MAX;
      for (int w = 0; w < kWarps; ++w) {
        // The warps' lists are sorted: merge each whole unless its best
        // cannot enter the top-ke.
        const int o = (w * QC + j) * 32;
        const float cs = ws[o + lane];
        const int ci = wi[o + lane];
        const float bs = __shfl_sync(kFullMask, cs, 0);
        const int bi = __shfl_sync(kFullMask, ci, 0);
        if (bi != INT_MAX && better(bs, bi, fs, fi)) {
          F.merge32(cs, ci);
          F.kth(ke, fs, fi);
        }
      }
      const int64_t pidx = a.part_off[done.g] + (int64_t)done.s * done.cg + done.q0 + j;
      if (lane == 0) a.part_ml[pidx] = make_float2(M, Ls);
      if (lane < ke) {
        a.part_s[pidx * ke + lane] = F.s0;
        a.part_id[pidx * ke + lane] = F.i0;
      }
    }
  }
  cp_async_wait<0>();
}

template <int QC, int KV>
htam_status launch_qk(const StreamArgs &a, int sm_count, cudaStream_t st) {
  const size_t smem = (size_t)kWarps * ring_slots<QC, KV>() * 32 * KV * 16 + side_bytes(QC);
  auto kernel = fine_ring_kernel<QC, KV>;
  HTAM_CK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  launch_kernel(kernel, sm_count, kWarps * 32, smem, st, a);
  HTAM_CK_LAUNCH("fine_ring_kernel");
  return HTAM_OK;
}

template <int QC>
htam_status launch_q(const StreamArgs &a, int kv, int sm_count, cudaStream_t st) {
  switch (kv) {
    case 1: return launch_qk<QC, 1>(a, sm_count, st);
    case 2: return launch_qk<QC, 2>(a, sm_count, st);
    case 4: return launch_qk<QC, 4>(a, sm_count, st);
    case 8:
      if constexpr (QC * 8 <= kMaxQueryVecs) return launch_qk<QC, 8>(a, sm_count, st);
      break;
    case 16:
      if constexpr (QC * 16 <= kMaxQueryVecs) return launch_qk<QC, 16>(a, sm_count, st);
      break;
  }
  return HTAM_EINVAL;
}

}  // namespace

htam_status launch_fine_stream(const StreamArgs &a, int qc, htam_dtype dtype, int sm_count, cudaStream_t st) {
  if (dtype != HTAM_BF16 || a.d % 8 != 0 || a.seg_pages < 1 || a.seg_pages > kMaxSegPages || a.ke > 32) {
    return HTAM_EINVAL;
  }
  const int per_lane = (a.d / 8 + 31) / 32;  // 16-byte query slices per lane
  int kv = 1;
  while (kv < per_lane) kv *= 2;
  if (kv * qc > kMaxQueryVecs) return HTAM_EINVAL;
  switch (qc) {
    case 8: return launch_q<8>(a, kv, sm_count, st);
    case 4: return launch_q<4>(a, kv, sm_count, st);
    case 2: return launch_q<2>(a, kv, sm_count, st);
    case 1: return launch_q<1>(a, kv, sm_count, st);
  }
  return HTAM_EINVAL;
}

}  // namespace htam
