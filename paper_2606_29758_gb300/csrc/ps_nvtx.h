// NVTX range around each C-ABI call, so a profiler's timeline (and ncu's --nvtx filters) shows
// which library call launched which kernels. Header-only NVTX 3: without an attached tool the
// push and pop are no-ops.
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace psk {

struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

}  // namespace psk
