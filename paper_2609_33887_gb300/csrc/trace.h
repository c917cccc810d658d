// Host-side trace range around one C-ABI call: an NVTX push/pop pair
// (header-only NVTX3; a no-op unless a profiler or tracer is attached).
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace bd {

struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};

}  // namespace bd
