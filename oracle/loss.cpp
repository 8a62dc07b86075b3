// Oracle — TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// GRPO token loss and its gradient with respect to the logits, Sec. 3.1 Eqs. 1-3.
//
// Per token t of a kept rollout o_i (row z of the logits, sampled token y):
//   pi_theta(y) = softmax(z)_y, so log pi_theta(y) = z_y - log sum_v exp(z_v)     (Sec. 3.2,
//                 last paragraph: logits -> softmax over the vocabulary -> token probability)
//   rho_t = pi_theta / pi_old = exp(logp - old_logp)                             (Eq. 1)
//   surrogate = min(rho*A, clip(rho, 1-eps, 1+eps)*A)                            (Eq. 1)
//   the KL term: Eqs. 2-3 give its gradient with respect to log pi_theta as
//       beta*(pi_ref/pi_theta - 1) = beta*(exp(x) - 1), x = ref_logp - logp,
//   whose antiderivative (zero at x = 0) is the per-token estimate kl = exp(x) - x - 1; the
//   objective carries -beta*kl.
//   The loss is the negated objective, l_t = -(surrogate - beta*kl), weighted by w_t.
//   Gradient of l_t w.r.t. log pi_theta: g_t = -(c*rho*A + beta*(exp(x) - 1)), with the clip
//   indicator c = [A>=0][rho<=1+eps] + [A<0][rho>=1-eps] (Sec. 3.1, after Eq. 3), and
//   d log pi_theta(y) / d z_v = [v == y] - softmax(z)_v, so
//       dlogits[t, v] = w_t * g_t * ([v == y] - exp(z_v - lse)).
// Weights: token mean (w_t = 1/denom) or Eq. 1's mean over sequences of per-sequence token
// means (w_t = 1/(n_seq * |o_i|)).
// Everything is fp64; outputs are rounded once at the end (f32 or bf16, nearest-even).
#include <cmath>
#include <cstring>
#include <limits>
#include <vector>

#ifdef _OPENMP
#include <omp.h>
#endif

#include "oracle.h"

namespace {

double load_logit(const void* logits, int dtype, int64_t idx) {
  if (dtype == 0) return (double)static_cast<const float*>(logits)[idx];
  if (dtype == 2) return static_cast<const double*>(logits)[idx];
  const uint32_t bits = (uint32_t) static_cast<const uint16_t*>(logits)[idx] << 16;
  float f;
  std::memcpy(&f, &bits, sizeof f);
  return (double)f;
}

void store_grad(void* out, int dtype, int64_t idx, double v) {
  if (dtype == 0)
    static_cast<float*>(out)[idx] = (float)v;
  else
    static_cast<uint16_t*>(out)[idx] = oracle_round_bf16(v);
}

}  // namespace

// Round to the nearest bf16 (8 significant bits, exponent range of f32, subnormals down to
// 2^-133), ties to even, directly from fp64 (one rounding).
extern "C" uint16_t oracle_round_bf16(double x) {
  const uint16_t sign = std::signbit(x) ? 0x8000 : 0;
  if (std::isnan(x)) return sign | 0x7FC0;
  const double ax = std::fabs(x);
  if (std::isinf(ax)) return sign | 0x7F80;
  if (ax == 0.0) return sign;
  int e;
  std::frexp(ax, &e);  // ax = m * 2^e, m in [0.5, 1): leading bit has weight 2^(e-1)
  int q = e - 8;       // weight of the last of 8 significant bits
  if (q < -133) q = -133;
  const double units = std::nearbyint(std::ldexp(ax, -q));  // exact scaling; ties to even
  const double v = std::ldexp(units, q);
  if (v >= std::ldexp(1.0, 128)) return sign | 0x7F80;
  const float f = (float)v;  // exact: v has at most 8 significant bits
  uint32_t bits;
  std::memcpy(&bits, &f, sizeof bits);
  return sign | (uint16_t)((bits >> 16) & 0x7FFF);
}

extern "C" int oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
  return omp_get_max_threads();
#else
  (void)n;
  return 1;
#endif
}

extern "C" int oracle_loss(const void* logits, int logits_dtype, int64_t row_stride,
                           const int64_t* row_index, int64_t n_rows, int V, const int32_t* y,
                           const float* old_logp, const float* ref_logp, const float* adv,
                           const int32_t* row_rollout, float eps_low, float eps_high, float beta,
                           int agg_mode, int64_t denom_tokens, const int64_t* seq_off,
                           int64_t n_seq, void* dlogits, int dlogits_dtype, double* dlogits_f64,
                           double* logp_out, double* rho_out, double* row_loss_out,
                           double* loss_out, double* g_out) {
  if (n_rows < 0 || V < 1 || row_stride < V) return 1;
  if (agg_mode == 0 && denom_tokens <= 0) return 1;
  if (agg_mode == 1 && (seq_off == nullptr || n_seq <= 0)) return 1;
  const double nan = std::numeric_limits<double>::quiet_NaN();
  std::vector<double> row_loss(n_rows, 0.0);

#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t t = 0; t < n_rows; ++t) {
    const int64_t src = row_index ? row_index[t] : t;
    const int64_t base = src * row_stride;
    const int32_t yt = y[src];
    if (yt < 0 || yt >= V) {  // invalid token: documented zero row
      for (int v = 0; v < V; ++v) {
        if (dlogits) store_grad(dlogits, dlogits_dtype, t * (int64_t)V + v, 0.0);
        if (dlogits_f64) dlogits_f64[t * (int64_t)V + v] = 0.0;
      }
      if (logp_out) logp_out[t] = nan;
      if (rho_out) rho_out[t] = nan;
      if (g_out) g_out[t] = nan;
      row_loss[t] = 0.0;
      continue;
    }
    // log-sum-exp over the vocabulary.
    double m = -std::numeric_limits<double>::infinity();
    for (int v = 0; v < V; ++v) m = std::fmax(m, load_logit(logits, logits_dtype, base + v));
    double s = 0.0;
    for (int v = 0; v < V; ++v) s += std::exp(load_logit(logits, logits_dtype, base + v) - m);
    const double lse = m + std::log(s);
    const double logp = load_logit(logits, logits_dtype, base + yt) - lse;

    // Eq. 1: importance ratio, clipped surrogate and KL penalty.
    const double A = (double)adv[row_rollout[t]];
    const double rho = std::exp(logp - (double)old_logp[src]);
    const double lo = 1.0 - (double)eps_low;
    const double hi = 1.0 + (double)eps_high;
    const double clipped = std::fmin(std::fmax(rho, lo), hi);
    const double surrogate = std::fmin(rho * A, clipped * A);
    const double x = (double)ref_logp[src] - logp;
    const double kl = std::exp(x) - x - 1.0;
    const double ell = -(surrogate - (double)beta * kl);

    double w;
    if (agg_mode == 0) {
      w = 1.0 / (double)denom_tokens;
    } else {
      const int32_t r = row_rollout[t];
      w = 1.0 / ((double)n_seq * (double)(seq_off[r + 1] - seq_off[r]));
    }
    row_loss[t] = w * ell;

    // Eqs. 2-3: gradient bracket, negated for the loss.
    const bool c = (A >= 0.0 && rho <= hi) || (A < 0.0 && rho >= lo);
    const double g = -((c ? rho * A : 0.0) + (double)beta * (std::exp(x) - 1.0));
    for (int v = 0; v < V; ++v) {
      const double p = std::exp(load_logit(logits, logits_dtype, base + v) - lse);
      const double d = w * g * ((v == yt ? 1.0 : 0.0) - p);
      if (dlogits) store_grad(dlogits, dlogits_dtype, t * (int64_t)V + v, d);
      if (dlogits_f64) dlogits_f64[t * (int64_t)V + v] = d;
    }
    if (logp_out) logp_out[t] = logp;
    if (rho_out) rho_out[t] = rho;
    if (g_out) g_out[t] = g;
  }

  double total = 0.0;
  for (int64_t t = 0; t < n_rows; ++t) total += row_loss[t];
  if (row_loss_out)
    for (int64_t t = 0; t < n_rows; ++t) row_loss_out[t] = row_loss[t];
  if (loss_out) *loss_out = total;
  return 0;
}

// Per-token log-probability alone (the old- and reference-policy evaluations of Sec. 3.2: logits
// -> softmax over the vocabulary -> probability of the sampled token): logp = z_y - log sum exp z.
extern "C" int oracle_logp(const void* logits, int logits_dtype, int64_t row_stride,
                           const int64_t* row_index, int64_t n_rows, int V, const int32_t* y,
                           double* logp_out) {
  if (n_rows < 0 || V < 1 || row_stride < V) return 1;
  const double nan = std::numeric_limits<double>::quiet_NaN();
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t t = 0; t < n_rows; ++t) {
    const int64_t src = row_index ? row_index[t] : t;
    const int64_t base = src * row_stride;
    const int32_t yt = y[src];
    if (yt < 0 || yt >= V) {
      logp_out[t] = nan;
      continue;
    }
    double m = -std::numeric_limits<double>::infinity();
    for (int v = 0; v < V; ++v) m = std::fmax(m, load_logit(logits, logits_dtype, base + v));
    double s = 0.0;
    for (int v = 0; v < V; ++v) s += std::exp(load_logit(logits, logits_dtype, base + v) - m);
    logp_out[t] = load_logit(logits, logits_dtype, base + yt) - (m + std::log(s));
  }
  return 0;
}

// GSPO's sequence-level loss over the kept rollouts: the base-algorithm variant FastRL is
// combined with in its experiments (Sec. 1 and Sec. 4, "GSPO"), with the objective of Group
// Sequence Policy Optimization (Zheng et al., 2025) restated here.  Rows come grouped by sequence:
// sequence k owns rows [seq_row_off[k], seq_row_off[k+1]) and rollout seq_rollout[k].
//   log s_k = (1/L_k) * sum_{t in k} (logp_t - old_logp_t)          (length-normalised ratio)
//   l_k = -( min(s_k*A, clip(s_k, 1-eps_low, 1+eps_high)*A) - beta*(1/L_k)*sum_t kl_t )
//   loss = (1/n_seq) * sum_k l_k,  kl_t = exp(x_t) - x_t - 1,  x_t = ref_logp_t - logp_t
// Gradient: d loss / d logp_t = w_t*g_t with w_t = 1/(n_seq*L_k) and
//   g_t = -(c_k*s_k*A + beta*(exp(x_t) - 1)),  c_k = [A>=0][s_k<=1+eps_high] + [A<0][s_k>=1-eps_low],
// so dlogits[t, v] = w_t*g_t*([v == y] - softmax(z)_v), as for the token-level ratio.
// A sequence holding an invalid token (y outside [0, V)) has no ratio: s_k = NaN, l_k = 0 and its
// rows' dlogits are 0.  Empty sequences (L_k = 0) contribute nothing.
extern "C" int oracle_gspo_loss(const void* logits, int logits_dtype, int64_t row_stride,
                                const int64_t* row_index, int V, const int32_t* y,
                                const float* old_logp, const float* ref_logp, const float* adv,
                                const int32_t* seq_rollout, const int64_t* seq_row_off,
                                int64_t n_seq_rows, int64_t n_seq, float eps_low, float eps_high,
                                float beta, void* dlogits, int dlogits_dtype, double* dlogits_f64,
                                double* logp_out, double* seq_ratio_out, double* seq_loss_out,
                                double* loss_out, double* g_out) {
  if (V < 1 || row_stride < V || n_seq_rows < 0 || n_seq <= 0 || seq_row_off == nullptr)
    return 1;
  if (seq_row_off[0] != 0) return 1;
  for (int64_t k = 0; k < n_seq_rows; ++k)
    if (seq_row_off[k + 1] < seq_row_off[k]) return 1;
  const int64_t n_rows = seq_row_off[n_seq_rows];
  const double nan = std::numeric_limits<double>::quiet_NaN();
  std::vector<double> logp(n_rows), lse(n_rows);

  // Per-row log-sum-exp and log-probability (as in oracle_loss).
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t t = 0; t < n_rows; ++t) {
    const int64_t src = row_index ? row_index[t] : t;
    const int64_t base = src * row_stride;
    const int32_t yt = y[src];
    if (yt < 0 || yt >= V) {
      logp[t] = nan;
      lse[t] = nan;
      continue;
    }
    double m = -std::numeric_limits<double>::infinity();
    for (int v = 0; v < V; ++v) m = std::fmax(m, load_logit(logits, logits_dtype, base + v));
    double s = 0.0;
    for (int v = 0; v < V; ++v) s += std::exp(load_logit(logits, logits_dtype, base + v) - m);
    lse[t] = m + std::log(s);
    logp[t] = load_logit(logits, logits_dtype, base + yt) - lse[t];
  }

  const double lo = 1.0 - (double)eps_low;
  const double hi = 1.0 + (double)eps_high;
  std::vector<double> seq_loss(n_seq_rows, 0.0);
  std::vector<double> coef(n_rows, 0.0);  // w_t * g_t
  if (g_out)  // rows of a sequence without a ratio keep NaN
    for (int64_t t = 0; t < n_rows; ++t) g_out[t] = nan;
  for (int64_t k = 0; k < n_seq_rows; ++k) {
    const int64_t r0 = seq_row_off[k], r1 = seq_row_off[k + 1];
    const int64_t L = r1 - r0;
    if (seq_ratio_out) seq_ratio_out[k] = nan;
    if (L == 0) continue;
    double sum_lr = 0.0, sum_kl = 0.0;
    bool valid = true;
    for (int64_t t = r0; t < r1; ++t) {
      const int64_t src = row_index ? row_index[t] : t;
      if (std::isnan(logp[t])) valid = false;
      sum_lr += logp[t] - (double)old_logp[src];
      const double x = (double)ref_logp[src] - logp[t];
      sum_kl += std::exp(x) - x - 1.0;
    }
    if (!valid) continue;
    const double A = (double)adv[seq_rollout[k]];
    const double s = std::exp(sum_lr / (double)L);
    const double clipped = std::fmin(std::fmax(s, lo), hi);
    const double surrogate = std::fmin(s * A, clipped * A);
    seq_loss[k] = -(surrogate - (double)beta * sum_kl / (double)L) / (double)n_seq;
    if (seq_ratio_out) seq_ratio_out[k] = s;
    const bool c = (A >= 0.0 && s <= hi) || (A < 0.0 && s >= lo);
    const double w = 1.0 / ((double)n_seq * (double)L);
    for (int64_t t = r0; t < r1; ++t) {
      const int64_t src = row_index ? row_index[t] : t;
      const double x = (double)ref_logp[src] - logp[t];
      const double g = -((c ? s * A : 0.0) + (double)beta * (std::exp(x) - 1.0));
      coef[t] = w * g;
      if (g_out) g_out[t] = g;
    }
  }

#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t t = 0; t < n_rows; ++t) {
    const int64_t src = row_index ? row_index[t] : t;
    const int64_t base = src * row_stride;
    const int32_t yt = y[src];
    const bool ok = yt >= 0 && yt < V;
    for (int v = 0; v < V; ++v) {
      double d = 0.0;
      if (ok && coef[t] != 0.0) {
        const double p = std::exp(load_logit(logits, logits_dtype, base + v) - lse[t]);
        d = coef[t] * ((v == yt ? 1.0 : 0.0) - p);
      }
      if (dlogits) store_grad(dlogits, dlogits_dtype, t * (int64_t)V + v, d);
      if (dlogits_f64) dlogits_f64[t * (int64_t)V + v] = d;
    }
    if (logp_out) logp_out[t] = logp[t];
  }
  double total = 0.0;
  for (int64_t k = 0; k < n_seq_rows; ++k) total += seq_loss[k];
  if (seq_loss_out)
    for (int64_t k = 0; k < n_seq_rows; ++k) seq_loss_out[k] = seq_loss[k];
  if (loss_out) *loss_out = total;
  return 0;
}
