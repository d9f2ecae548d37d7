// fine_stream.h -- CUDA-core fine-score kernel for small buckets, with the
// entry rows streamed through shared memory by bulk asynchronous copies.
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
  unsigned *status;
  uint32_t max_polls;
};

// Rows up to this many bytes are streamed (a ring stage holds at least one).
constexpr int kStreamMaxRowBytes = 8192;

// Launches the streaming kernel for `qc` queries per unit (1, 2, 4 or 8) on
// bf16 or fp32 rows.  Returns HTAM_EINVAL without launching when the row is
// longer than a stage or the shared memory would not fit (the caller then
// uses the direct-load kernel).
htam_status launch_fine_stream(const StreamArgs &a, int qc, htam_dtype dtype, int sm_count, cudaStream_t st);

}  // namespace htam
