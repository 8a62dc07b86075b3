// NVTX ranges around the library's C-ABI calls that enqueue GPU work.  NVTX 3 is header-only: a
// range costs a few nanoseconds and records nothing unless a tool such as Nsight Compute or
// Nsight Systems is attached, which then attributes each kernel to its call (for instance
// `ncu --nvtx --nvtx-include "grpo_loss_fwd_bwd/"` profiles that call's kernels only).
#pragma once

#include <nvtx3/nvToolsExt.h>

namespace fastrl {

class TraceRange {
 public:
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};

}  // namespace fastrl

#define GRPO_TRACE(name) ::fastrl::TraceRange grpo_trace_range_(name)
