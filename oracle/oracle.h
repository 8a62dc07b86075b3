/*
 * Reference oracle for the FastRL kept-token GRPO path — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, fp64 CPU restatement of what the path computes, written from the paper's
 * definitions ("Learn from the Gap", Sec. 3 and Algorithm 1).  Only the test suite, the smoke
 * check and the benchmark's CPU-baseline leg may load it.  It shares no code, header, table or
 * helper with the CUDA library: nothing here includes or links anything from the package, and
 * the package never loads this.
 *
 * Every function follows one passage of the paper; the pins that check each one against what
 * the paper and the mathematics fix live in tests/test_oracle_*.py.  Floating point is fp64
 * throughout, on inputs given in f32 or as bf16 bit patterns (both exact in fp64).  Build with
 * -ffp-contract=off so that no multiply-add is fused: advantages and pruning keys are then
 * reproducible bit for bit from their written order of operations.
 */
#ifndef FASTRL_ORACLE_H_
#define FASTRL_ORACLE_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Eq. 5: per-group advantages; see advantage.cpp. */
int oracle_advantage(const float* rewards, int P, int G, int std_mode, float* adv, double* key);

/* Eqs. 6-9 and Algorithm 1 (Phase 2 and DP alignment): MDAP keep mask; see mdap.cpp. */
int oracle_prune(const float* rewards, const int32_t* ids, const int64_t* off, int P, int G,
                 int ngram_n, float tau, int keep_cap, int dp_divisor, uint8_t* keep,
                 int32_t* kept_per_prompt);

/* The same with the continuous-reward grouping: class_eps > 0 groups rollouts whose advantages
 * (adv, f32 [P*G]) chain with consecutive sorted gaps below class_eps. */
int oracle_prune_classes(const float* rewards, const float* adv, float class_eps,
                         const int32_t* ids, const int64_t* off, int P, int G, int ngram_n,
                         float tau, int keep_cap, int dp_divisor, uint8_t* keep,
                         int32_t* kept_per_prompt);

/* Eq. 7 alone, for tests: theta_ij for rollouts i and j (indices into off). */
double oracle_jaccard_distance(const int32_t* ids, const int64_t* off, int i, int j, int ngram_n);

/* Compaction of kept rollouts' tokens (Sec. 3.2 after Eq. 9); see compact.cpp. */
int oracle_compact(const uint8_t* keep, const int64_t* off, int n_rollouts, int32_t* kept_idx,
                   int64_t* kept_off, int64_t* src_token, int32_t* token_rollout, int64_t* counts);

/* Eqs. 1-3: GRPO token loss and dlogits; see loss.cpp.
 * logits_dtype 0 = f32, 1 = bf16 bit patterns (uint16), 2 = f64.  dlogits_dtype 0 = f32,
 * 1 = bf16 bits.
 * dlogits_f64 (nullable) receives the unrounded fp64 gradient.  rho_out (nullable) the ratios.
 * g_out (nullable) each row's g_t = -(c*rho*A + beta*(exp(x) - 1)), the factor that multiplies
 * w_t*([v == y] - softmax_v) in its dlogits (NaN for an invalid token). */
int oracle_loss(const void* logits, int logits_dtype, int64_t row_stride, const int64_t* row_index,
                int64_t n_rows, int V, const int32_t* y, const float* old_logp,
                const float* ref_logp, const float* adv, const int32_t* row_rollout, float eps_low,
                float eps_high, float beta, int agg_mode, int64_t denom_tokens,
                const int64_t* seq_off, int64_t n_seq, void* dlogits, int dlogits_dtype,
                double* dlogits_f64, double* logp_out, double* rho_out, double* row_loss_out,
                double* loss_out, double* g_out);

/* GSPO's sequence-level loss (length-normalised sequence ratio, clipped per sequence) over kept
 * rollouts; see loss.cpp.  Sequence k owns rows [seq_row_off[k], seq_row_off[k+1]) of the
 * n_seq_rows sequences and rollout seq_rollout[k]; loss = (1/n_seq) sum_k l_k.
 * seq_ratio_out [n_seq_rows] (nullable): s_k (NaN when undefined); seq_loss_out: l_k / n_seq.
 * g_out [rows] (nullable): each row's gradient factor g_t = -(c_k s_k A + beta (exp(x_t) - 1)),
 * dlogits[t] = g_t / (n_seq L_k) * (onehot(y) - softmax); NaN in a sequence without a ratio. */
int oracle_gspo_loss(const void* logits, int logits_dtype, int64_t row_stride,
                     const int64_t* row_index, int V, const int32_t* y, const float* old_logp,
                     const float* ref_logp, const float* adv, const int32_t* seq_rollout,
                     const int64_t* seq_row_off, int64_t n_seq_rows, int64_t n_seq, float eps_low,
                     float eps_high, float beta, void* dlogits, int dlogits_dtype,
                     double* dlogits_f64, double* logp_out, double* seq_ratio_out,
                     double* seq_loss_out, double* loss_out, double* g_out);

/* The policy's output layer fused with the GRPO token loss; see lmhead.cpp.
 * hidden f64 [n_rows, D], weight f64 [V, D] (row-major; bf16 values widen exactly).
 * z = hidden * weight^T, then oracle_loss on z (Eqs. 1-3), then the chain rule:
 * dhidden = dlogits * weight [n_rows, D], dweight = dlogits^T * hidden [V, D].
 * Every output is nullable.  dhidden_abs / dweight_abs receive the same products over absolute
 * values (|dlogits| * |weight|, |dlogits|^T * |hidden|), the scale of the rounding error of any
 * evaluation of dhidden and dweight. */
int oracle_lmhead_loss(const double* hidden, const double* weight, int64_t n_rows, int V, int D,
                       const int32_t* y, const float* old_logp, const float* ref_logp,
                       const float* adv, const int32_t* row_rollout, float eps_low,
                       float eps_high, float beta, int agg_mode, int64_t denom_tokens,
                       const int64_t* seq_off, int64_t n_seq, double* logits_out,
                       double* dlogits_out, double* logp_out, double* row_loss_out,
                       double* loss_out, double* dhidden, double* dweight, double* dhidden_abs,
                       double* dweight_abs);

/* The same with GSPO's sequence-level ratio: oracle_gspo_loss on z = hidden * weight^T (sequences
 * as oracle_gspo_loss takes them, over the n_rows rows), then the chain rule.  Nullable outputs. */
int oracle_lmhead_gspo_loss(const double* hidden, const double* weight, int64_t n_rows, int V,
                            int D, const int32_t* y, const float* old_logp, const float* ref_logp,
                            const float* adv, const int32_t* seq_rollout,
                            const int64_t* seq_row_off, int64_t n_seq_rows, int64_t n_seq,
                            float eps_low, float eps_high, float beta, double* dlogits_out,
                            double* logp_out, double* seq_ratio_out, double* seq_loss_out,
                            double* loss_out, double* dhidden, double* dweight,
                            double* dhidden_abs, double* dweight_abs);

/* logp of the sampled token alone (old/reference policy evaluation); NaN for ids outside [0,V). */
int oracle_logp(const void* logits, int logits_dtype, int64_t row_stride, const int64_t* row_index,
                int64_t n_rows, int V, const int32_t* y, double* logp_out);

/* Round an fp64 value to bf16 (nearest, ties to even, bf16 subnormals kept); returns the bits. */
uint16_t oracle_round_bf16(double x);

/* Eqs. 10-14 and Algorithm 1 (Phases 1a/1b): adaptive rollout sampling; see ars.cpp. */
void* oracle_ars_new(int G1);
void oracle_ars_free(void* st);
int oracle_ars_step(void* st, const int32_t* kept_per_prompt, int P, int64_t step,
                    int64_t total_steps, int epoch_end);
double oracle_ars_get(void* st, int what); /* 0: G'_ref or NaN, 1: G'_t or NaN */

/* Worker threads the loss uses (OpenMP); 0 keeps the runtime default.  Returns the count. */
int oracle_set_threads(int n);

/* The chain rule through z = hidden * weight^T alone, for given fp64 dlogits [n_rows, V]:
 * dhidden = dlogits * weight, dweight = dlogits^T * hidden (each nullable), and the sums of the
 * absolute products (nullable); see lmhead.cpp. */
int oracle_lmhead_grad(const double* hidden, const double* weight, const double* dlogits,
                       int64_t n_rows, int V, int D, double* dhidden, double* dweight,
                       double* dhidden_abs, double* dweight_abs);

#ifdef __cplusplus
}
#endif

#endif /* FASTRL_ORACLE_H_ */
