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
// count, nullable), min(n, *n_dev); one launch of an 8-CTA cluster on `s`, as a programmatic
// dependent of the kernel before it (its reads wait for that kernel to complete).
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

// Bytes of dynamic shared memory this launch was given.
__device__ __forceinline__ uint32_t dynamic_smem_bytes() {
  uint32_t n;
  asm("mov.u32 %0, %%dynamic_smem_size;" : "=r"(n));
  return n;
}

// Programmatic dependent launch (PTX griddepcontrol).  When every CTA of a kernel has called
// allow_dependent_launch() (or exited), the next kernel of the stream, if it was launched with
// cudaLaunchAttributeProgrammaticStreamSerialization, may be scheduled before the first one ends;
// that kernel calls wait_for_prerequisite_grids() before its first global access, which returns
// once the earlier grid has completed and its writes are visible.  A kernel launched without the
// attribute returns from the wait at once.
__device__ __forceinline__ void allow_dependent_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void wait_for_prerequisite_grids() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---- index checks of the checked build -----------------------------------------------------
// build.py's checked build (libfastrl_grpo_checked.so) compiles every file with GRPO_CHECKED:
// GRPO_DCHECK(cond) then evaluates cond where a kernel is about to read or write through an
// index it computed (a gathered row, a shared-memory slot, a copy's address and size, a tile
// coordinate); a false cond records this file (GRPO_TU) and the first failing source line in
// the file's device flags, and the caller skips the access.  grpo_debug_checks reads and clears
// the flags.  In the normal build GRPO_DCHECK(cond) is `true` and cond is not evaluated.
#if defined(GRPO_CHECKED)
#ifndef GRPO_TU
#error "each file defines GRPO_TU (its index in grpo_debug_checks' mask) before common.cuh"
#endif
namespace {
__device__ int32_t g_dcheck_mask;  // one pair per file (anonymous namespace)
__device__ int32_t g_dcheck_site;
__device__ __forceinline__ bool dcheck(bool ok, int line) {
  if (!ok) {
    atomicOr(&g_dcheck_mask, 1 << GRPO_TU);
    atomicCAS(&g_dcheck_site, 0, GRPO_TU * 100000 + line);
  }
  return ok;
}
}  // namespace
#define GRPO_DCHECK(cond) ::fastrl::dcheck(static_cast<bool>(cond), __LINE__)
// Defines `grpo_status name(bool reset, int32_t* mask, int32_t* site)` for this file's flags
// (on the current device; the caller has synchronised it).
#define GRPO_DCHECK_READER(name)                                                        \
  grpo_status name(bool reset, int32_t* mask, int32_t* site) {                          \
    int32_t m = 0, st = 0;                                                              \
    if (cudaMemcpyFromSymbol(&m, g_dcheck_mask, sizeof(m)) != cudaSuccess ||            \
        cudaMemcpyFromSymbol(&st, g_dcheck_site, sizeof(st)) != cudaSuccess)            \
      return GRPO_ERR_CUDA;                                                             \
    *mask |= m;                                                                         \
    if (*site == 0) *site = st;                                                         \
    if (reset) {                                                                        \
      const int32_t z = 0;                                                              \
      if (cudaMemcpyToSymbol(g_dcheck_mask, &z, sizeof(z)) != cudaSuccess ||            \
          cudaMemcpyToSymbol(g_dcheck_site, &z, sizeof(z)) != cudaSuccess)              \
        return GRPO_ERR_CUDA;                                                           \
    }                                                                                   \
    return GRPO_OK;                                                                     \
  }
grpo_status dcheck_read_advantage(bool, int32_t*, int32_t*);
grpo_status dcheck_read_prune(bool, int32_t*, int32_t*);
grpo_status dcheck_read_compact(bool, int32_t*, int32_t*);
grpo_status dcheck_read_loss(bool, int32_t*, int32_t*);
grpo_status dcheck_read_gspo(bool, int32_t*, int32_t*);
grpo_status dcheck_read_reduce(bool, int32_t*, int32_t*);
grpo_status dcheck_read_lmhead(bool, int32_t*, int32_t*);
grpo_status dcheck_read_gemm(bool, int32_t*, int32_t*);
#else
#define GRPO_DCHECK(cond) true
#define GRPO_DCHECK_READER(name)
#endif

}  // namespace fastrl
