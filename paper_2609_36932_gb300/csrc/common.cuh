// Shared host and device helpers of libfastrl_grpo (CUDA path only).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "fastrl_grpo.h"

namespace fastrl {

// ---- host side -------------------------------------------------------------------------------

// Record a message for grpo_last_error() and return `s`.
grpo_status fail(grpo_status s, const char* fmt, ...);
// Clear the calling thread's message.
void clear_error();
// Count `n` kernel launches (grpo_kernel_launches()).
void count_launches(uint64_t n);
// Check the last launch; on failure record `what` and return GRPO_ERR_CUDA.
grpo_status check_launch(const char* what);

inline cudaStream_t as_stream(grpo_stream_t s) { return reinterpret_cast<cudaStream_t>(s); }

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace protocol: ws == NULL -> report `need` in *ws_bytes; otherwise check the size.
grpo_status workspace_check(void* ws, size_t* ws_bytes, size_t need, const char* who,
                            bool* query_only);

// ---- device side -----------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

}  // namespace fastrl
