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

// Forward-only row kernel (loss.cu): logp_out[t] = z_y - log sum_v exp(z_v) for n_rows rows, or
// min(n_rows, counts[1]) with device counts {K, T_kept} (rows and errors as grpo_logp_fwd) and,
// with stats_out, each row's softmax statistics {max M, sum of exp(z - M), that sum without y, 0}
// (NaN for a token id outside [0, V)).
grpo_status logp_rows(const char* who, const void* logits, int32_t logits_dtype, int64_t row_stride,
                      const int64_t* row_index, int64_t n_rows, const int64_t* counts, int32_t V,
                      const int32_t* y, float* logp_out, float4* stats_out, int32_t* status,
                      cudaStream_t s);

// reduce.cu: *out = v[0] + ... + v[m-1] in fp64 in a fixed order, m = n or, with n_dev (a device
// count, nullable), min(n, *n_dev); one launch of an 8-CTA cluster on `s`.
grpo_status launch_sum_rows(const double* v, int64_t n, const int64_t* n_dev, double* out,
                            cudaStream_t s, const char* who);

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
