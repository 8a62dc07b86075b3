// Oracle — TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// Adaptive rollout sampling (ARS), Sec. 3.3 Eqs. 10-14, in the step order of Algorithm 1:
//   Phase 1(b), after pruning a step: append G'^mean_t = mean_q |S(q)| and G'^max_t = max_q |S(q)|
//     (Eq. 10) to two epoch buffers.  At an epoch boundary, alpha = step / total_steps and
//     G'_t = alpha * mean(B_mean) + (1 - alpha) * mean(B_max) (Eq. 11); after the first epoch,
//     G'_ref = (mean(B_mean) + mean(B_max)) / 2 (Eq. 12); then both buffers are emptied.
//   Phase 1(a), before the next step: if G'_t and G'_ref are both set and G'_t < G'_ref,
//     Delta = G'_ref - G'_t (Eq. 13) and n = max(round(min(G_1 - Delta, G_1)), 2) (Eq. 14);
//     otherwise n = G_1.
// round() is read as round-half-to-even (the rounding of the Python frameworks the paper uses).
#include <cmath>
#include <limits>
#include <vector>

#include "oracle.h"

namespace {

struct ArsOracle {
  int G1 = 0;
  int n = 0;
  bool have_ref = false;
  bool have_gt = false;
  double g_ref = 0.0;
  double g_t = 0.0;
  std::vector<double> b_mean;
  std::vector<double> b_max;
};

double average(const std::vector<double>& b) {
  double s = 0.0;
  for (double v : b) s += v;
  return s / (double)b.size();
}

}  // namespace

extern "C" void* oracle_ars_new(int G1) {
  ArsOracle* st = new ArsOracle();
  st->G1 = G1;
  st->n = G1;
  return st;
}

extern "C" void oracle_ars_free(void* st) { delete static_cast<ArsOracle*>(st); }

extern "C" double oracle_ars_get(void* p, int what) {
  const ArsOracle* st = static_cast<ArsOracle*>(p);
  const double nan = std::numeric_limits<double>::quiet_NaN();
  if (what == 0) return st->have_ref ? st->g_ref : nan;
  return st->have_gt ? st->g_t : nan;
}

extern "C" int oracle_ars_step(void* p, const int32_t* kept_per_prompt, int P, int64_t step,
                               int64_t total_steps, int epoch_end) {
  ArsOracle* st = static_cast<ArsOracle*>(p);
  if (P < 1 || step < 1 || total_steps < step) return -1;
  // Eq. 10.
  long sum = 0;
  int mx = kept_per_prompt[0];
  for (int q = 0; q < P; ++q) {
    sum += kept_per_prompt[q];
    if (kept_per_prompt[q] > mx) mx = kept_per_prompt[q];
  }
  st->b_mean.push_back((double)sum / (double)P);
  st->b_max.push_back((double)mx);
  if (epoch_end) {
    const double alpha = (double)step / (double)total_steps;
    const double mean_bar = average(st->b_mean);
    const double max_bar = average(st->b_max);
    st->g_t = alpha * mean_bar + (1.0 - alpha) * max_bar;  // Eq. 11
    st->have_gt = true;
    if (!st->have_ref) {
      st->g_ref = (mean_bar + max_bar) / 2.0;  // Eq. 12
      st->have_ref = true;
    }
    st->b_mean.clear();
    st->b_max.clear();
  }
  // Eqs. 13-14.
  if (st->have_gt && st->have_ref && st->g_t < st->g_ref) {
    const double delta = st->g_ref - st->g_t;
    const double target = std::fmin((double)st->G1 - delta, (double)st->G1);
    const int rounded = (int)std::nearbyint(target);
    st->n = rounded > 2 ? rounded : 2;
  } else {
    st->n = st->G1;
  }
  return st->n;
}
