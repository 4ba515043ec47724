// NVTX range around one C-ABI call, so that a timeline profiler shows each
// entry point's host-side span (argument checks and kernel enqueue, not the
// kernels' device time) under the entry point's name. With no profiler
// attached the NVTX calls return at once. Host code only.
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace smetric {

class CallRange {
 public:
  explicit CallRange(const char* name) { nvtxRangePushA(name); }
  ~CallRange() { nvtxRangePop(); }
  CallRange(const CallRange&) = delete;
  CallRange& operator=(const CallRange&) = delete;
};

}  // namespace smetric
