// Fixed-order fp64 sum of per-row (or per-sequence) loss terms: the last step of every loss call
// and of grpo_sum_f64, so that a loss computed in one call or in chunks sums to the same bits.
//
// One CTA of 1024 threads.  Thread t adds v[t], v[t + 1024], v[t + 2048], ... in that order,
// loading kBatch of them before adding any (the loads overlap; the order of the additions does
// not change); then a fixed xor-shuffle tree inside each warp and one more across the 32 warps.
#include "common.cuh"
#include "trace.cuh"

namespace fastrl {
namespace {

constexpr int kSumThreads = 1024;
constexpr int kBatch = 8;

__global__ void __launch_bounds__(kSumThreads)
    sum_rows_kernel(const double* __restrict__ v, int64_t n, const int64_t* __restrict__ n_dev,
                    double* __restrict__ out) {
  __shared__ double part[kSumThreads / 32];
  if (n_dev && *n_dev < n) n = *n_dev;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  double acc = 0.0;
  for (int64_t base = tid; base < n; base += (int64_t)kSumThreads * kBatch) {
    double x[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int64_t i = base + (int64_t)u * kSumThreads;
      x[u] = i < n ? v[i] : 0.0;
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) acc += x[u];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) part[warp] = acc;
  __syncthreads();
  if (warp == 0) {
    acc = part[lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) *out = acc;
  }
}

}  // namespace

grpo_status launch_sum_rows(const double* v, int64_t n, const int64_t* n_dev, double* out,
                            cudaStream_t s, const char* who) {
  sum_rows_kernel<<<1, kSumThreads, 0, s>>>(v, n, n_dev, out);
  count_launches(1);
  return check_launch(who);
}

}  // namespace fastrl

using namespace fastrl;

extern "C" grpo_status grpo_sum_f64(const double* v, int64_t n, double* out, grpo_stream_t stream) {
  GRPO_TRACE("grpo_sum_f64");
  clear_error();
  if (n < 0 || out == nullptr || (n > 0 && v == nullptr))
    return fail(GRPO_ERR_INVALID_ARG, "grpo_sum_f64: n = %lld, v or out NULL", (long long)n);
  return launch_sum_rows(v, n, nullptr, out, as_stream(stream), "grpo_sum_f64");
}
