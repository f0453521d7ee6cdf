// validate.cuh -- host-side argument checks shared by the entry points of
// api.cu and compact.cu (internal header): every entry point that takes a
// batch or a gather list accepts exactly the same ones.
#pragma once

#include <stdint.h>

#include "occam.h"

namespace occam {

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The batch descriptor's sizes and pointers (device arrays are not read).
inline int check_batch(const occam_batch* b) {
  if (!b) return OCCAM_ERR_INVALID_ARG;
  if (b->B < 1 || b->S_tot < b->B || b->total_rows < 1 || b->total_rows >= (int64_t(1) << 31) ||
      b->total_text < 0 || b->total_text >= (int64_t(1) << 31) || b->max_seg_rows < 1 ||
      b->max_sample_rows < b->max_seg_rows || b->max_text < 0 || b->max_regs < 1)
    return OCCAM_ERR_INVALID_ARG;
  if (!b->row_off || !b->seg_off || !b->seg_first || !b->seg_sample || !b->reg_idx || !b->reg_off ||
      !b->text_off)
    return OCCAM_ERR_INVALID_ARG;
  return OCCAM_OK;
}

// A gather list of n row tensors: 16-byte aligned bases and row sizes.
inline int check_gather(int n, const void* const* src, const int64_t* rb, void* const* dst) {
  if (n < 0 || n > OCCAM_MAX_GATHER) return OCCAM_ERR_INVALID_ARG;
  for (int t = 0; t < n; ++t) {
    if (!src || !dst || !rb || !src[t] || !dst[t] || rb[t] <= 0 || (rb[t] & 15) || !aligned16(src[t]) ||
        !aligned16(dst[t]))
      return OCCAM_ERR_INVALID_ARG;
  }
  return OCCAM_OK;
}

}  // namespace occam
