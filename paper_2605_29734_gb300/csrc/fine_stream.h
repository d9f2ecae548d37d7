// fine_stream.h -- CUDA-core fine-score kernel for small buckets, with the
// entry rows prefetched into per-warp shared-memory rings by cp.async.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "htam.h"

namespace htam {

struct StreamArgs {
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
  const int4 *units;          // (group, bucket chunk, page segment)
  const int32_t *n_units;
  const int64_t *part_off;
  int ke;
  float inv_tau;
  int seg_pages;
  float2 *part_ml;
  float *part_s;
  int32_t *part_id;
};

// Every ring holds at least this many rows per warp (two in flight while the
// third is scored).
constexpr int kStreamMinSlots = 3;

// Launches the ring kernel for `qc` queries per unit (1, 2, 4 or 8) on bf16
// rows.  Returns HTAM_EINVAL without launching for fp32 rows, for
// k_entries > 32, or when the unit's queries do not fit in 128 registers
// per lane, i.e. for rows longer than 8 KiB (the caller then uses the
// direct-load kernel).
htam_status launch_fine_stream(const StreamArgs &a, int qc, htam_dtype dtype, int sm_count, cudaStream_t st);

}  // namespace htam
