// bsm_trace.h -- NVTX ranges around the host entry points (plan creation and
// execution, the host-buffer pipeline), so that they show up by name on a
// profiler's timeline next to the kernels they launch.  NVTX v3 is
// header-only; without a profiler attached every call is a no-op.
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace bsm {

struct TraceRange {
    explicit TraceRange(const char *name) { nvtxRangePushA(name); }
    ~TraceRange() { nvtxRangePop(); }
    TraceRange(const TraceRange &) = delete;
    TraceRange &operator=(const TraceRange &) = delete;
};

}  // namespace bsm
