// check.cuh -- in-kernel bounds checks of the checked build (internal
// header). Built with -DOCCAM_CHECKED=1, every computed index at the sites
// below is tested against the extent of the buffer it addresses before the
// access; the first violation writes OCCAM_ERR_BOUNDS to the status word and
// its site number to the word after it, and the access is skipped or
// redirected to a valid row. Nothing traps or asserts. In the default build
// the checks compile to nothing.
#pragma once

#ifndef OCCAM_CHECKED
#define OCCAM_CHECKED 0
#endif

namespace occam {

// check sites (the status word's companion word names the first that failed)
enum CheckSite {
  kSiteGatherRow = 1,      // gather: the source row of an output position
  kSiteStageRow = 2,       // staging: an S1 row id
  kSiteScanSample = 3,     // scan: the sample of a tile's first row
  kSiteLogitsSegment = 4,  // Stage-I logits: the segment of a row
  kSiteListPos = 5,        // Stage-I finalize: a position in the sample's S1 list
  kSiteRegisterRow = 6,    // Stage-I finalize: a register row of the segment
  kSiteFusedItem = 7,      // fused Stage II: a work item's sample and text tile
  kSiteFusedKeyRow = 8,    // fused Stage II: an S1 key row (TMA gather coordinate)
  kSiteFusedSlot = 9,      // fused Stage II: an s2(r) partial slot
  kSiteTwoPassKeyRow = 10, // two-pass Stage II: an S1 key row
  kSiteMutualRow = 11,     // mutual Stage I: a row of the segment
};

// True when ok; otherwise (checked builds) records the first violation and
// returns false. status: the call's status word (int32 [2]).
__device__ __forceinline__ bool in_bounds(bool ok, int* status, int site) {
#if OCCAM_CHECKED
  if (!ok && status && atomicCAS(status, 0, 7 /* OCCAM_ERR_BOUNDS */) == 0) atomicExch(status + 1, site);
  return ok;
#else
  (void)status;
  (void)site;
  return true;
#endif
}

}  // namespace occam
