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
// fp64 throughout; the dlogits that enter the chain rule are the loss oracle's unrounded ones.
// With GSPO's sequence-level ratio (Sec. 1, Sec. 4) the middle step is oracle_gspo_loss instead.
#include <cmath>
#include <vector>

#include "oracle.h"

namespace {

// z[t, v] = sum_d h[t, d] * W[v, d]: one dot product per (token, vocabulary entry).
void output_layer(const double* hidden, const double* weight, int64_t n_rows, int V, int D,
                  std::vector<double>& z) {
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
}

// The chain rule through z = h W^T, each sum over v or t in increasing order (the loops are
// arranged to read memory in order).
void chain_rule(const double* hidden, const double* weight, int64_t n_rows, int V, int D,
                const std::vector<double>& dl, double* dhidden, double* dweight,
                double* dhidden_abs, double* dweight_abs) {
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
}

void copy_out(const std::vector<double>& src, int64_t n, double* dst) {
  if (dst)
    for (int64_t i = 0; i < n; ++i) dst[i] = src[i];
}

}  // namespace

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
  output_layer(hidden, weight, n_rows, V, D, z);
  copy_out(z, nz, logits_out);

  // Eqs. 1-3 on those logits.
  std::vector<double> dl(nz > 0 ? nz : 1);
  std::vector<double> logp(n_rows > 0 ? n_rows : 1), rho(n_rows > 0 ? n_rows : 1);
  std::vector<double> rl(n_rows > 0 ? n_rows : 1);
  double total = 0.0;
  const int rc = oracle_loss(z.data(), 2, V, nullptr, n_rows, V, y, old_logp, ref_logp, adv,
                             row_rollout, eps_low, eps_high, beta, agg_mode, denom_tokens, seq_off,
                             n_seq, nullptr, 0, dl.data(), logp.data(), rho.data(), rl.data(),
                             &total, nullptr);
  if (rc != 0) return rc;
  copy_out(dl, nz, dlogits_out);
  copy_out(logp, n_rows, logp_out);
  copy_out(rl, n_rows, row_loss_out);
  if (loss_out) *loss_out = total;
  chain_rule(hidden, weight, n_rows, V, D, dl, dhidden, dweight, dhidden_abs, dweight_abs);
  return 0;
}

extern "C" int oracle_lmhead_gspo_loss(const double* hidden, const double* weight, int64_t n_rows,
                                       int V, int D, const int32_t* y, const float* old_logp,
                                       const float* ref_logp, const float* adv,
                                       const int32_t* seq_rollout, const int64_t* seq_row_off,
                                       int64_t n_seq_rows, int64_t n_seq, float eps_low,
                                       float eps_high, float beta, double* dlogits_out,
                                       double* logp_out, double* seq_ratio_out,
                                       double* seq_loss_out, double* loss_out, double* dhidden,
                                       double* dweight, double* dhidden_abs, double* dweight_abs) {
  if (n_rows < 0 || V < 1 || D < 1) return 1;
  const int64_t nz = n_rows * (int64_t)V;
  std::vector<double> z(nz > 0 ? nz : 1);
  output_layer(hidden, weight, n_rows, V, D, z);

  // GSPO's sequence-level loss on those logits.
  std::vector<double> dl(nz > 0 ? nz : 1);
  std::vector<double> logp(n_rows > 0 ? n_rows : 1);
  double total = 0.0;
  const int rc = oracle_gspo_loss(z.data(), 2, V, nullptr, V, y, old_logp, ref_logp, adv,
                                  seq_rollout, seq_row_off, n_seq_rows, n_seq, eps_low, eps_high,
                                  beta, nullptr, 0, dl.data(), logp.data(), seq_ratio_out,
                                  seq_loss_out, &total, nullptr);
  if (rc != 0) return rc;
  copy_out(dl, nz, dlogits_out);
  copy_out(logp, n_rows, logp_out);
  if (loss_out) *loss_out = total;
  chain_rule(hidden, weight, n_rows, V, D, dl, dhidden, dweight, dhidden_abs, dweight_abs);
  return 0;
}

// The chain rule alone, for dlogits given in fp64: dh = dlogits * W and dW = dlogits^T * h, with
// the sums of absolute products (the error bound's scale) when asked for.
extern "C" int oracle_lmhead_grad(const double* hidden, const double* weight, const double* dlogits,
                                  int64_t n_rows, int V, int D, double* dhidden, double* dweight,
                                  double* dhidden_abs, double* dweight_abs) {
  if (n_rows < 0 || V < 1 || D < 1) return 1;
  const int64_t nz = n_rows * (int64_t)V;
  std::vector<double> dl(dlogits, dlogits + nz);
  chain_rule(hidden, weight, n_rows, V, D, dl, dhidden, dweight, dhidden_abs, dweight_abs);
  return 0;
}
