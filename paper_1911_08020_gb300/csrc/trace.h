// trace.h -- NVTX ranges around the C-ABI calls, so that a profiler's timeline
// (Nsight Systems, Nsight Compute's NVTX filters) shows which library call
// enqueued which kernels and how long the host part of each call took.  NVTX3
// is header-only: with no tool attached a range costs a check of a function
// pointer; a tool is attached through the NVTX_INJECTION64_PATH environment
// variable, read once at the first range of the process.
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace darb {

struct TraceRange {
    explicit TraceRange(const char *name) { nvtxRangePushA(name); }
    ~TraceRange() { nvtxRangePop(); }
    TraceRange(const TraceRange &) = delete;
    TraceRange &operator=(const TraceRange &) = delete;
};

}  // namespace darb

// One range named after the enclosing C-ABI call, from here to its return.
#define DARB_TRACE(name) const ::darb::TraceRange darb_trace_range_(name)
