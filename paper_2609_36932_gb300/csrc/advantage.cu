// grpo_advantage: group-relative advantages, Eq. 5 (Sec. 3.2).
//
// One warp per prompt.  The fp64 sums run in index order (every lane executes the same
// sequence of explicitly rounded additions on values exchanged by shuffles), so the mean, the
// std and each A are reproducible bit for bit from the order of operations written here; the
// per-rollout divisions then run in parallel across lanes.
#define GRPO_TU 0  // this file's bit in the checked build's report (grpo_debug_checks)
#include "common.cuh"
#include "trace.cuh"

namespace fastrl {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__global__ void advantage_kernel(const float* __restrict__ rewards, int P, int G, int std_mode,
                                 float* __restrict__ adv, double* __restrict__ key) {
  const int p = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (p >= P) return;  // uniform per warp
  const float* r = rewards + (int64_t)p * G;
  double sum = 0.0;
  for (int base = 0; base < G; base += 32) {
    const float v = base + lane < G ? r[base + lane] : 0.f;
    const int nb = min(32, G - base);
    for (int k = 0; k < nb; ++k) sum = __dadd_rn(sum, (double)__shfl_sync(kFull, v, k));
  }
  const double mean = __ddiv_rn(sum, (double)G);
  double ss = 0.0;
  for (int base = 0; base < G; base += 32) {
    const float v = base + lane < G ? r[base + lane] : 0.f;
    const double dev = __dsub_rn((double)v, mean);
    const double sq = __dmul_rn(dev, dev);
    const int nb = min(32, G - base);
    for (int k = 0; k < nb; ++k) ss = __dadd_rn(ss, __shfl_sync(kFull, sq, k));
  }
  const int divisor = std_mode == 0 ? G - 1 : G;
  const double sd = divisor > 0 ? __dsqrt_rn(__ddiv_rn(ss, (double)divisor)) : 0.0;
  for (int i = lane; i < G; i += 32) {
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
  GRPO_TRACE("grpo_advantage");
  clear_error();
  if (P < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: P = %d < 0", P);
  if (G < 1 || G > 1024) return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: G = %d not in [1, 1024]", G);
  if (std_mode != 0 && std_mode != 1)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: std_mode = %d not 0 or 1", std_mode);
  if (P == 0) return GRPO_OK;
  if (rewards == nullptr || adv == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_advantage: rewards and adv must not be NULL");
  const int threads = 128;  // four prompts per CTA
  advantage_kernel<<<(unsigned)(((int64_t)P * 32 + threads - 1) / threads), threads, 0, as_stream(stream)>>>(
      rewards, P, G, std_mode, adv, key);
  count_launches(1);
  return check_launch("grpo_advantage");
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_advantage)
}  // namespace fastrl
