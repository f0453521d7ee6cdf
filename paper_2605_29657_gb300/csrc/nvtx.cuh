// NVTX ranges on the host timeline, one per launch group of the prune path
// (Stage I scores, Stage I threshold, the staging copy, Stage II scores, the
// Stage II threshold and the compaction / gather), nested in one range per
// C-ABI call, all in the "occam" domain. Nsight tools attach to them (ncu
// --nvtx --nvtx-include "occam@occam_prune/", nsys); without an attached tool
// a push or pop returns at once. Compiled out with -DOCCAM_NVTX=0.
#pragma once

#ifndef OCCAM_NVTX
#define OCCAM_NVTX 1
#endif

#if OCCAM_NVTX
#include <nvtx3/nvToolsExt.h>

namespace occam_nvtx {
inline nvtxDomainHandle_t domain() {
  static nvtxDomainHandle_t d = nvtxDomainCreateA("occam");
  return d;
}
}  // namespace occam_nvtx

struct NvtxRange {
  explicit NvtxRange(const char* name) {
    nvtxEventAttributes_t a = {};
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    nvtxDomainRangePushEx(occam_nvtx::domain(), &a);
  }
  ~NvtxRange() { nvtxDomainRangePop(occam_nvtx::domain()); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};
#else
struct NvtxRange {
  explicit NvtxRange(const char*) {}
};
#endif
