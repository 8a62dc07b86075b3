// The output layer's backward products on the tensor cores (gemm.cu), for lmhead.cu.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "fastrl_grpo.h"

namespace fastrl {

// How gemm_bf16 runs a product: K split into S ranges of kb_per 64-wide blocks, `units` work
// units of a 256 x 256 tile over one range, on `grid` CTAs; partial_bytes of f32 workspace for
// the S partial products when S > 1.
struct GemmPlan {
  int S, kb_per, units, grid;
  size_t partial_bytes;
};
GemmPlan gemm_plan(int64_t M, int64_t N, int64_t K, int n_sm);

// C[m, n] = sum_k A(m, k) * B(k, n) (+ C[m, n] with accumulate), bf16 A and B, f32 accumulation
// on the tensor cores; C f32 or bf16 (c_dtype), row stride ldc >= N.  B is stored [K][N] (row
// stride ldb).  A is stored [M][K] (a_mn false) or [K][M] (a_mn true), row stride lda.  lda and
// ldb are multiples of 8, A and B 16-byte aligned, N a multiple of 4; accumulate needs f32 C.
// `partial` (nullable, 16-byte aligned) is the workspace for a split K (gemm_plan's
// partial_bytes); without it the product runs unsplit.  Asynchronous on `s`; GRPO_DEVFLAG_TIMEOUT
// in *status (nullable) if a bounded wait ran out.
grpo_status gemm_bf16(const char* who, bool a_mn, const void* A, int64_t lda, const void* B,
                      int64_t ldb, int64_t M, int64_t N, int64_t K, void* C, int64_t ldc,
                      int32_t c_dtype, bool accumulate, float* partial, size_t partial_bytes,
                      int32_t* status, cudaStream_t s);

}  // namespace fastrl
