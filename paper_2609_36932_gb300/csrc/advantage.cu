// grpo_advantage: group-relative advantages, Eq. 5 (Sec. 3.2).
//
// One thread per prompt.  A group has at most a few dozen rewards, so the fp64 sums run
// sequentially in index order with explicitly rounded operations (no fused multiply-add); the
// result is then reproducible bit for bit from the order of operations written here.
#include "common.cuh"

namespace fastrl {
namespace {

__global__ void advantage_kernel(const float* __restrict__ rewards, int P, int G, int std_mode,
                                 float* __restrict__ adv, double* __restrict__ key) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= P) return;
  const float* r = rewards + (int64_t)p * G;
  double sum = 0.0;
  for (int i = 0; i < G; ++i) sum = __dadd_rn(sum, (double)r[i]);
  const double mean = __ddiv_rn(sum, (double)G);
  double ss = 0.0;
  for (int i = 0; i < G; ++i) {
    const double dev = __dsub_rn((double)r[i], mean);
    ss = __dadd_rn(ss, __dmul_rn(dev, dev));
  }
  const int divisor = std_mode == 0 ? G - 1 : G;
  const double sd = divisor > 0 ? __dsqrt_rn(__ddiv_rn(ss, (double)divisor)) : 0.0;
  for (int i = 0; i < G; ++i) {
    const double dev = __dsub_rn((double)r[i], mean);
    const double a = sd > 0.0 ? __ddiv_rn(dev, sd) : 0.0;
    adv[(int64_t)p * G + i] = __double2float_rn(a);
    if (key) key[(int64_t)p * G + i] = fabs(dev);
  }
}

}  // namespace
}  // namespace fastrl

using namespace fastrl;

extern "C" grpo_status grpo_advantage(const float* rewards, int32_t P, int32_t G, int32_t std_mode,
                                      float* adv, double* key, grpo_stream_t stream) {
  clear_error();
  if (P < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: P = %d < 0", P);
  if (G < 1 || G > 1024) return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: G = %d not in [1, 1024]", G);
  if (std_mode != 0 && std_mode != 1)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: std_mode = %d not 0 or 1", std_mode);
  if (P == 0) return GRPO_OK;
  if (rewards == nullptr || adv == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: rewards and adv must not be NULL");
  const int threads = 128;
  advantage_kernel<<<(P + threads - 1) / threads, threads, 0, as_stream(stream)>>>(
      rewards, P, G, std_mode, adv, key);
  count_launches(1);
  return check_launch("grpo_advantage");
}
