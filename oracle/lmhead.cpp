// Oracle — TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// The policy's output layer fused with the GRPO token loss.  Sec. 3.2 runs the kept trajectories
// through the policy, whose last layer turns each token's hidden state into logits over the
// vocabulary before the softmax; Eqs. 1-3 then give the loss.  With hidden states h[t, :] (D
// values per kept token) and the output layer's weight rows W[v, :]:
//   z[t, v] = sum_d h[t, d] * W[v, d]                       (the logits, never rounded here)
//   loss, logp, dlogits = oracle_loss on z                  (Eqs. 1-3, in loss.cpp)
//   dh[t, d] = sum_v dlogits[t, v] * W[v, d]                (chain rule through z = h W^T)
//   dW[v, d] = sum_t dlogits[t, v] * h[t, d]
// fp64 throughout; the dlogits that enter the chain rule are oracle_loss's unrounded ones.
#include <cmath>
#include <vector>

#include "oracle.h"

extern "C" int oracle_lmhead_loss(const double* hidden, const double* weight, int64_t n_rows,
                                  int V, int D, const int32_t* y, const float* old_logp,
                                  const float* ref_logp, const float* adv,
                                  const int32_t* row_rollout, float eps_low, float eps_high,
                                  float beta, int agg_mode, int64_t denom_tokens,
                                  const int64_t* seq_off, int64_t n_seq, double* logits_out,
                                  double* dlogits_out, double* logp_out, double* row_loss_out,
                                  double* loss_out, double* dhidden, double* dweight,
                                  double* dhidden_abs, double* dweight_abs) {
  if (n_rows < 0 || V < 1 || D < 1) return 1;
  const int64_t nz = n_rows * (int64_t)V;
  std::vector<double> z(nz > 0 ? nz : 1);

  // The output layer: one dot product per (token, vocabulary entry).
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t t = 0; t < n_rows; ++t) {
    const double* h = hidden + t * D;
    for (int v = 0; v < V; ++v) {
      const double* w = weight + (int64_t)v * D;
      double acc = 0.0;
      for (int d = 0; d < D; ++d) acc += h[d] * w[d];
      z[t * V + v] = acc;
    }
  }
  if (logits_out)
    for (int64_t i = 0; i < nz; ++i) logits_out[i] = z[i];

  // Eqs. 1-3 on those logits.
  std::vector<double> dl(nz > 0 ? nz : 1);
  std::vector<double> logp(n_rows > 0 ? n_rows : 1), rho(n_rows > 0 ? n_rows : 1);
  std::vector<double> rl(n_rows > 0 ? n_rows : 1);
  double total = 0.0;
  const int rc = oracle_loss(z.data(), 2, V, nullptr, n_rows, V, y, old_logp, ref_logp, adv,
                             row_rollout, eps_low, eps_high, beta, agg_mode, denom_tokens, seq_off,
                             n_seq, nullptr, 0, dl.data(), logp.data(), rho.data(), rl.data(),
                             &total);
  if (rc != 0) return rc;
  if (dlogits_out)
    for (int64_t i = 0; i < nz; ++i) dlogits_out[i] = dl[i];
  if (logp_out)
    for (int64_t t = 0; t < n_rows; ++t) logp_out[t] = logp[t];
  if (row_loss_out)
    for (int64_t t = 0; t < n_rows; ++t) row_loss_out[t] = rl[t];
  if (loss_out) *loss_out = total;

  // Chain rule through z = h W^T: with respect to the hidden states ...  (each sum runs over v
  // or t in increasing order; the loops are arranged to read memory in order)
  if (dhidden || dhidden_abs) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t t = 0; t < n_rows; ++t) {
      std::vector<double> acc(D, 0.0), aabs(D, 0.0);
      for (int v = 0; v < V; ++v) {
        const double g = dl[t * V + v];
        const double* w = weight + (int64_t)v * D;
        for (int d = 0; d < D; ++d) {
          acc[d] += g * w[d];
          aabs[d] += std::fabs(g) * std::fabs(w[d]);
        }
      }
      for (int d = 0; d < D; ++d) {
        if (dhidden) dhidden[t * D + d] = acc[d];
        if (dhidden_abs) dhidden_abs[t * D + d] = aabs[d];
      }
    }
  }
  // ... and with respect to the weight.
  if (dweight || dweight_abs) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int v = 0; v < V; ++v) {
      std::vector<double> acc(D, 0.0), aabs(D, 0.0);
      for (int64_t t = 0; t < n_rows; ++t) {
        const double g = dl[t * V + v];
        const double* h = hidden + t * D;
        for (int d = 0; d < D; ++d) {
          acc[d] += g * h[d];
          aabs[d] += std::fabs(g) * std::fabs(h[d]);
        }
      }
      for (int d = 0; d < D; ++d) {
        if (dweight) dweight[(int64_t)v * D + d] = acc[d];
        if (dweight_abs) dweight_abs[(int64_t)v * D + d] = aabs[d];
      }
    }
  }
  return 0;
}
