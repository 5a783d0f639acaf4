// trace.h -- a named NVTX range around each C-ABI entry point, for timeline tools (Nsight Systems,
// ncu --nvtx).  NVTX v3 is header-only; a range costs a few nanoseconds when no tool is attached.
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace wino {

struct Range {
    explicit Range(const char *name) { nvtxRangePushA(name); }
    ~Range() { nvtxRangePop(); }
    Range(const Range &) = delete;
    Range &operator=(const Range &) = delete;
};

}  // namespace wino
