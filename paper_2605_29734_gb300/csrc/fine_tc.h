// fine_tc.h -- tensor-core (tcgen05) fine-score kernel of the lookup.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "htam.h"

namespace htam {

constexpr int kTcRows = 128;      // queries per tensor-core work unit (MMA M)
constexpr int kTcMaxK = 32;       // largest k_entries the tensor-core path keeps

// Per-query shared score bounds of the tensor-core units: word 0 is the best
// k-th score any unit's own list has reached; word 1 + s is the best
// ceil(k / kThrSlots)-th score of the units whose page segment index is s
// modulo kThrSlots.  Units of different classes hold disjoint entries, so
// kThrSlots * ceil(k / kThrSlots) >= k candidates score at least the smallest
// of those words: both are lower bounds of the query's final k-th best score.
constexpr int kThrSlots = 4;
constexpr int kThrWords = 1 + kThrSlots;

struct TcFineArgs {
  const int4 *units;          // (group, bucket chunk, page segment)
  const int32_t *n_units;     // device count of units
  int32_t *unit_ctr;          // units taken beyond the first per CTA; zero before the launch
  const int32_t *bucket;      // bucket rows -> query id
  const int32_t *bucket_off;  // [G+1]
  const int32_t *cnt;         // [G] bucket sizes
  const int32_t *page_list;
  const int32_t *page_off;
  const int32_t *count;       // [G] entries per group
  const int32_t *slot_id;
  const int64_t *part_off;
  int d;
  const int32_t *seg_pages;  // device: pages per unit (even), chosen by the bucketing
  int ke;
  float k2;                   // log2(e) / tau
  float2 *part_ml;
  float *part_s;
  int32_t *part_id;
  unsigned *thr_enc;          // [B][kThrWords] order-preserving encodings of the shared bounds above
  unsigned *status;           // memory status word
  uint32_t max_polls;
  int q_direct;               // 1: every bucket holds all queries in order and the query map is the
                              // query matrix itself (rows from 0), 0: rows from bucket_off[g]
  // a_rows = 1 (one-SM units): a copier warp copies each chunk's query rows
  // from the query matrix `queries` (`qvec` 16-byte vectors a row) with
  // cp.async into the swizzled A stages; the query map is then unused.
  // 0: the A tiles come from the query map by TMA.
  int a_rows;
  const uint4 *queries;
  int qvec;
};

// Encodes a 2-D bf16 row-major [rows, cols] tensor for TMA tile loads of
// box {64 columns, box_rows rows} with the 128-byte swizzle.
htam_status make_bf16_tile_map(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols,
                               uint32_t box_rows);

// Queries gathered into bucket order, as the A operand of the kernel.
htam_status launch_gather_queries(const void *Q, int d, const int32_t *bucket, const int32_t *bucket_group,
                                  const int32_t *cnt, int tc_min, const int32_t *total_rows, int64_t max_rows,
                                  void *Qg, cudaStream_t st);

// pair: the units are (group, pair of 128-query chunks, segment), run by
// clusters of two CTAs (grid rounded down to even); otherwise (group, chunk,
// segment), one CTA each.
htam_status launch_fine_tc(const TcFineArgs &a, const CUtensorMap &q_map, const CUtensorMap &pool_map, int grid,
                           bool pair, cudaStream_t st);

}  // namespace htam
