/*
 * fastrl_grpo.h — C ABI of the GB300 kept-token GRPO library (libfastrl_grpo.so).
 *
 * The library computes, on one GPU, the data-parallel core of one FastRL training step
 * ("Learn from the Gap", Sec. 3 and Algorithm 1):
 *
 *   grpo_advantage          group-relative advantages                  (Eq. 5)
 *   grpo_prune              maximising-differential advantage pruning  (Eqs. 6-9, Algorithm 1)
 *   grpo_compact            compaction of the kept rollouts' tokens    (Sec. 3.2, after Eq. 9)
 *   grpo_loss_fwd_bwd       fused GRPO token loss and dlogits          (Eqs. 1-3)
 *     (_dev: row count read on the device, for CUDA graphs; _noalloc: no workspace)
 *   grpo_logp_fwd           log-probabilities alone                    (Sec. 3.2)
 *   grpo_gspo_loss_fwd_bwd  GSPO's sequence-level loss                 (Sec. 1, Sec. 4)
 *     (_dev: counts read on the device, for CUDA graphs)
 *   grpo_lmhead_loss_fwd_bwd  the output layer fused with the loss:     (Sec. 3.2, Eqs. 1-3)
 *                           logits on the tensor cores, one chunk of rows at a time; dhidden,
 *                           dweight
 *     (grpo_lmhead_logp_fwd: log-probabilities alone from hidden states;
 *      grpo_lmhead_gspo_loss_fwd_bwd: the same with GSPO's sequence-level loss;
 *      grpo_lmhead_grad: dhidden and dweight from given dlogits)
 *   grpo_upload_kept        host-to-device copy of the kept rows only  (Sec. 3.2)
 *   adaptive_rollout_count  adaptive rollout sampling, on the host     (Eqs. 10-14, Algorithm 1)
 *
 * Conventions shared by every call:
 *   - Every call returns a grpo_status; GRPO_OK is 0.  On failure, grpo_last_error() returns a
 *     message for the calling thread.  No C++ exception and no abort crosses this boundary.
 *   - Buffers marked "device" are device pointers owned by the caller (for instance memory held
 *     by PyTorch tensors).  The library never allocates or frees device memory, with one
 *     exception: grpo_loss_fwd_bwd_noalloc's fixed 2 MiB scratch array, which every GPU that
 *     loads the library holds until the process exits.  Scratch memory otherwise
 *     comes from a caller workspace: a call with ws == NULL and ws_bytes != NULL only writes the
 *     size it needs into *ws_bytes and enqueues nothing.  The real call passes ws (256-byte
 *     aligned) with *ws_bytes >= that size, or ws == NULL and ws_bytes == NULL when the size
 *     is 0.
 *   - GPU work is enqueued asynchronously on `stream` (a cudaStream_t; NULL is the legacy
 *     default stream).  Host-side argument errors are returned before anything is enqueued.
 *   - Data errors that only the GPU can see (a token id outside [0, V), non-finite logits, a
 *     wait that ran out of time) never trap: kernels OR a GRPO_DEVFLAG_* bit into the caller's
 *     int32 device status word, which the caller reads after synchronising the stream.
 *   - All arrays are dense and row-major unless a stride argument says otherwise.
 */
#ifndef FASTRL_GRPO_H_
#define FASTRL_GRPO_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef void* grpo_stream_t; /* a cudaStream_t */

typedef enum {
  GRPO_OK = 0,
  GRPO_ERR_INVALID_ARG = 1,  /* a null pointer, a negative size or an out-of-range parameter */
  GRPO_ERR_UNSUPPORTED = 2,  /* a valid request outside this build's limits (stated per call) */
  GRPO_ERR_WORKSPACE = 3,    /* workspace missing or smaller than the size query returned */
  GRPO_ERR_CUDA = 4,         /* a CUDA runtime call failed; grpo_last_error() names it */
  GRPO_ERR_TIMEOUT = 5,      /* a device wait ran out (grpo_check_status on a status word) */
  GRPO_ERR_DEVICE_CHECK = 6  /* a kernel flagged bad data (grpo_check_status on a status word) */
} grpo_status;

typedef enum { GRPO_DTYPE_F32 = 0, GRPO_DTYPE_BF16 = 1 } grpo_dtype;

/* Bits a kernel ORs into the caller's device status word. */
#define GRPO_DEVFLAG_BAD_TOKEN 1 /* a token id outside [0, V) */
#define GRPO_DEVFLAG_NONFINITE 2 /* a row's log-sum-exp or log-prob was NaN or infinite */
#define GRPO_DEVFLAG_TIMEOUT 4   /* a bounded wait on an asynchronous copy gave up */

/* Message describing the last failure on the calling thread ("" if none). */
const char* grpo_last_error(void);

/* Library version string. */
const char* grpo_version(void);

/* Number of kernels this process has launched through the library so far (host counter). */
uint64_t grpo_kernel_launches(void);

/*
 * grpo_debug_checks — the report of the checked build's device index checks (no counterpart in
 * the paper; a stand-in for a memory checker, which this library's GPUs do not offer).  The
 * checked build (libfastrl_grpo_checked.so, same ABI) tests, inside its kernels, every index it
 * computes before reading or writing through it: gathered rows, shared-memory slots, the address,
 * size and alignment of each asynchronous copy, tile coordinates and output extents.  A failing
 * check skips that access and records its source file and line; nothing traps.
 * Synchronises the current device, then sets *file_mask to the files whose checks failed since
 * the last reset (bit i: advantage.cu 0, prune.cu 1, compact.cu 2, loss.cu 3, gspo.cu 4,
 * reduce.cu 5, lmhead.cu 6, gemm.cu 7) and *first_site to 100000 * file + line of a first
 * failure (0 if none); reset != 0 clears the record.  The normal build returns
 * GRPO_ERR_UNSUPPORTED with both outputs 0; grpo_version() names the checked build.
 */
grpo_status grpo_debug_checks(int32_t reset, int32_t* file_mask, int32_t* first_site);

/*
 * grpo_check_status — turn a device status word, read back by the caller after synchronising
 * the stream its kernels ran on, into a grpo_status (host only, no GPU work; no counterpart in
 * the paper).  0 gives GRPO_OK.  GRPO_DEVFLAG_TIMEOUT gives GRPO_ERR_TIMEOUT: a bounded wait
 * gave up and that launch's results are invalid.  Otherwise any bit (GRPO_DEVFLAG_BAD_TOKEN,
 * GRPO_DEVFLAG_NONFINITE, unknown bits) gives GRPO_ERR_DEVICE_CHECK: the flagged rows have the
 * documented NaN log-prob / zero gradient and the other rows are valid.  grpo_last_error() then
 * names every bit that is set.
 */
grpo_status grpo_check_status(int32_t status_word);

/*
 * grpo_advantage — group-relative advantage, Eq. 5 (Sec. 3.2):
 *   A_i = (r_i - mean{r_1..r_G}) / std{r_1..r_G}, one group of G rollouts per prompt.
 * rewards   device f32 [P*G], prompt-major (rollout i of prompt p at p*G + i).
 * std_mode  0: sample std (divide by G-1); 1: population std (divide by G).
 * adv       device f32 [P*G] out.  A group whose std is 0 (all rewards equal), or G == 1 in
 *           mode 0, gets A = 0.  mean and std are taken in fp64, summed in index order, and
 *           A is rounded once to f32.
 * key       device f64 [P*G] out, nullable: |r_i - mean| in fp64, the ordering key MDAP uses.
 * Limits: 1 <= G <= 1024.  P = 0 is a no-op.
 */
grpo_status grpo_advantage(const float* rewards, int32_t P, int32_t G, int32_t std_mode,
                           float* adv, double* key, grpo_stream_t stream);

/*
 * grpo_prune — maximising-differential advantage pruning, Eqs. 6-9 and Algorithm 1 (Phase 2).
 * Per prompt q, rollouts are partitioned into classes of equal advantage (Eq. 6); inside a
 * group A is a strictly increasing function of r, so classes are taken by exact f32 reward
 * equality.  Rollouts are visited by |r_i - mean| descending (fp64), ties by lower index, and
 * a rollout is kept unless an already kept rollout of its class has Jaccard distance
 * theta_ij = 1 - |N_n(o_i) & N_n(o_j)| / |N_n(o_i) | N_n(o_j)| < tau (Eqs. 7-8), where N_n is
 * the set of distinct n-grams of a completion.  Two rollouts that both have no n-gram
 * (length < n) have theta = 0.  The kept set is S(q), the union over classes (Eq. 9).
 * Then, if |S(q)| > keep_cap, keep_cap rollouts are kept by round-robin over the classes
 * (classes ordered by the visiting position of their first member; each round takes each
 * class's next kept rollout in visiting order, which for equal rewards is the lowest index).
 * keep_cap >= G disables the cap (the paper's rule).  Finally, while the total kept count is
 * not a multiple of dp_divisor, prompts are visited cyclically from prompt 0 and each visit adds
 * that prompt's unkept rollout with the largest |r - mean| (lowest index on ties); prompts with
 * none left are skipped (Algorithm 1, DP alignment).  dp_divisor = 1 does nothing.
 * rewards          device f32 [P*G].
 * adv, class_eps   class_eps = 0: classes by exact reward equality (adv may be NULL).
 *                  class_eps > 0: the continuous-reward grouping of the paper's grounding
 *                  extension, |A_i - A_j| < class_eps (the paper uses 1e-4), closed under
 *                  transitivity: with the advantages adv (device f32 [P*G], e.g. grpo_advantage's)
 *                  sorted ascending (ties by index), a new class starts wherever the gap to the
 *                  previous value is >= class_eps (differences in fp64).
 * ids              device i32 [T]: completion token ids of all rollouts, packed.
 * off              device i64 [P*G+1]: rollout r owns ids[off[r] .. off[r+1]); off[0] = 0,
 *                  off[P*G] = T, non-decreasing.
 * ngram_n          1..3.  Token ids must lie in [0, V); an id outside it sets
 *                  GRPO_DEVFLAG_BAD_TOKEN and leaves that prompt's keep mask unspecified.
 * tau              Jaccard-distance threshold (the paper uses 0.8).
 * keep_cap         >= 1, per-prompt cap after MDAP.
 * dp_divisor       >= 1.
 * keep             device u8 [P*G] out: 1 = kept.
 * kept_per_prompt  device i32 [P] out: |S(q)| after cap and fill.
 * status           device i32 [1], nullable: GRPO_DEVFLAG_* bits are ORed in.
 * ws, ws_bytes     workspace (see conventions); its size depends on T, P and G.
 * Limits: 1 <= G <= 32; 1 <= V <= 2^18 (three 18-bit ids fit one 64-bit n-gram key).
 */
grpo_status grpo_prune(const float* rewards, const float* adv, float class_eps, const int32_t* ids,
                       const int64_t* off, int32_t P, int32_t G, int64_t T, int32_t V,
                       int32_t ngram_n, float tau, int32_t keep_cap, int32_t dp_divisor,
                       uint8_t* keep, int32_t* kept_per_prompt, int32_t* status, void* ws,
                       size_t* ws_bytes, grpo_stream_t stream);

/*
 * grpo_compact — token compaction of the kept rollouts (Sec. 3.2: only retained trajectories
 * are fed to the old, current and reference models).
 * keep           device u8 [n_rollouts].
 * off            device i64 [n_rollouts+1] token offsets of all rollouts.
 * kept_idx       device i32 [n_rollouts] out: indices of the K kept rollouts, ascending.
 * kept_off       device i64 [n_rollouts+1] out: kept_off[k] = tokens of kept rollouts before k;
 *                kept_off[K] = T_kept.
 * src_token      device i64 [T] out: for kept row t < T_kept, its token index in `off` layout.
 * token_rollout  device i32 [T] out: for kept row t < T_kept, its rollout index (0..n_rollouts).
 * counts         device i64 [2] out: {K, T_kept}.
 * counts_host    host i64 [2], nullable: if given, {K, T_kept} are copied there (a stream-ordered
 *                copy; use pinned memory and synchronise the stream before reading).
 * Entries past K (kept_idx, kept_off) and past T_kept (src_token, token_rollout) are untouched.
 */
grpo_status grpo_compact(const uint8_t* keep, const int64_t* off, int32_t n_rollouts,
                         int32_t* kept_idx, int64_t* kept_off, int64_t* src_token,
                         int32_t* token_rollout, int64_t* counts, int64_t* counts_host,
                         grpo_stream_t stream);

/*
 * grpo_upload_kept — host-to-device transfer of the kept rollouts' token rows only.  Sec. 3.2
 * feeds only the retained trajectories to the models, so a step whose per-token inputs (for
 * instance logits) live in host memory need not move the pruned rollouts' rows at all.
 * For every maximal run of consecutive kept rollouts i..j (keep_host[r] != 0) one
 * cudaMemcpyAsync on `stream` copies bytes [off_host[i]*row_bytes, off_host[j+1]*row_bytes) of
 * src_host to the same offset of dst_dev.  Rows of pruned rollouts in dst_dev are not written.
 * src_host   host, token rows of row_bytes bytes in `off_host` layout.  Pinned memory makes the
 *            copies asynchronous; the runtime copies pageable memory synchronously.
 * dst_dev    device, the same layout and size.
 * keep_host  host u8 [n_rollouts] (grpo_prune's keep, copied back); off_host host i64
 *            [n_rollouts+1], off_host[0] >= 0 and non-decreasing.
 * bytes_out, copies_out  host, nullable: bytes and copies enqueued.
 * Errors (before any copy is enqueued): GRPO_ERR_INVALID_ARG for a NULL array with
 * n_rollouts > 0, n_rollouts < 0, row_bytes <= 0, decreasing or negative offsets, or a byte
 * offset that overflows int64.  GRPO_ERR_CUDA if a copy cannot be enqueued (copies enqueued
 * before it stay enqueued).  No kernel is launched.
 */
grpo_status grpo_upload_kept(const void* src_host, void* dst_dev, int64_t row_bytes,
                             const uint8_t* keep_host, const int64_t* off_host,
                             int32_t n_rollouts, int64_t* bytes_out, int32_t* copies_out,
                             grpo_stream_t stream);

/*
 * grpo_loss_fwd_bwd — fused GRPO token loss and its gradient w.r.t. the logits, Eqs. 1-3.
 * For every row t < n_rows, with z the logits row, y the sampled token and A the advantage:
 *   lse = log sum_v exp(z_v);  logp = z_y - lse;  rho = exp(logp - old_logp)
 *   surr = min(rho*A, clip(rho, 1-eps_low, 1+eps_high)*A)
 *   x = ref_logp - logp;  kl = exp(x) - x - 1                      (per-token KL estimate)
 *   l_t = -(surr - beta*kl);  loss = sum_t w_t * l_t
 *   c = [A>=0][rho<=1+eps_high] + [A<0][rho>=1-eps_low]             (clip indicator, Sec. 3.1)
 *   g_t = -(c*rho*A + beta*(exp(x) - 1))                            (bracket of Eq. 3, negated)
 *   dlogits[t, v] = w_t * g_t * ([v == y] - exp(z_v - lse))
 * Weights: agg_mode 0 (token mean): w_t = 1/denom_tokens.  agg_mode 1 (Eq. 1's sequence mean):
 *   w_t = 1/(n_seq * L_r), L_r = seq_off[r+1] - seq_off[r] for the row's rollout r.
 * Inputs:
 *   logits        device, dtype logits_dtype (GRPO_DTYPE_BF16 or GRPO_DTYPE_F32); row s starts
 *                 at element s*row_stride (row_stride >= V).
 *   row_index     device i64 [n_rows], nullable: row t reads logits row src = row_index[t]
 *                 (for instance grpo_compact's src_token); if NULL, src = t.
 *   y, old_logp, ref_logp   device i32 / f32 / f32, indexed by src.
 *   adv           device f32 advantage per rollout; row_rollout device i32 [n_rows] gives the
 *                 rollout of row t (indexed by t, for instance grpo_compact's token_rollout).
 *   eps_low, eps_high  clip range; beta >= 0 the KL weight.
 *   denom_tokens  > 0 in agg_mode 0 (for data parallelism: the global kept-token count).
 *   seq_off, n_seq  used in agg_mode 1 only (device i64 rollout offsets, host count > 0).
 * Outputs (indexed by t):
 *   dlogits       device [n_rows, V] contiguous, dtype dlogits_dtype, rounded to nearest even.
 *   logp_out      device f32 [n_rows], nullable.
 *   row_loss_out  device f64 [n_rows], nullable: w_t * l_t.
 *   loss_out      device f64 [1]: the sum, reduced in a fixed order (bitwise reproducible).
 *   status        device i32 [1], nullable: GRPO_DEVFLAG_* bits.  A row whose y lies outside
 *                 [0, V) gets logp = NaN, a zero dlogits row and a zero loss term.
 * Workspace: n_rows f64 when row_loss_out is NULL, else none.
 * Limits: V >= 1, V*element size <= 16 * 200 KiB; n_rows < 2^31.
 * Alignment: logits and dlogits must be aligned to their element size (else
 *   GRPO_ERR_INVALID_ARG).  Rows need not start on a 16-byte boundary, but such rows are slower:
 *   logits rows that do start on one arrive by bulk copies, and dlogits rows by 16-byte stores;
 *   other rows (an odd V stored densely, such as 50257) are realigned by the kernel, which
 *   measured about 3.5 TB/s with both sides unaligned at V = 50257 and about 4.6 TB/s with only
 *   the dlogits rows unaligned, against 5.9 TB/s aligned (V = 50264), with the same bits as an
 *   aligned call on the same values.  Padding the vocabulary to a multiple of 8 with -inf logits
 *   gives the same results on the true columns (exp(-inf) = 0 in every sum) and zero dlogits
 *   (+0 or -0) on the padding.
 */
grpo_status grpo_loss_fwd_bwd(const void* logits, int32_t logits_dtype, int64_t row_stride,
                              const int64_t* row_index, int64_t n_rows, int32_t V,
                              const int32_t* y, const float* old_logp, const float* ref_logp,
                              const float* adv, const int32_t* row_rollout, float eps_low,
                              float eps_high, float beta, int32_t agg_mode, int64_t denom_tokens,
                              const int64_t* seq_off, int64_t n_seq, void* dlogits,
                              int32_t dlogits_dtype, float* logp_out, double* row_loss_out,
                              double* loss_out, int32_t* status, void* ws, size_t* ws_bytes,
                              grpo_stream_t stream);

/*
 * grpo_logp_fwd — log-probability of the sampled token alone, for the old- and reference-policy
 * evaluations over the kept trajectories (Sec. 3.2: the retained trajectories go through the old,
 * current and reference models; logits -> softmax over the vocabulary -> token probability):
 *   logp_out[t] = z_y - log sum_v exp(z_v),  z = logits row src, y = y[src], src = row_index[t]
 *   (or t when row_index is NULL).  One read of the logits, no gradient, no loss.
 * logits, row_stride, row_index, y: as grpo_loss_fwd_bwd.  logp_out device f32 [n_rows].
 * status: device i32, nullable (GRPO_DEVFLAG_BAD_TOKEN leaves logp = NaN, GRPO_DEVFLAG_NONFINITE).
 * Limits: as grpo_loss_fwd_bwd.  No workspace.
 * Alignment: as grpo_loss_fwd_bwd.  Rows that do not start on a 16-byte boundary are realigned
 *   (two aligned 16-byte loads per vector), with the same bits as an aligned call: about 4.2 TB/s
 *   against 7.0 at V = 152064.
 * Kernel: one CTA streams each row (no cluster, no shared-memory slice; grpo_loss_tune does not
 * apply).  Its sums run in a different order from the fused loss's, so the two log-probabilities
 * agree to within a few ulps, not bit for bit; each is deterministic.
 */
grpo_status grpo_logp_fwd(const void* logits, int32_t logits_dtype, int64_t row_stride,
                          const int64_t* row_index, int64_t n_rows, int32_t V, const int32_t* y,
                          float* logp_out, int32_t* status, grpo_stream_t stream);

/*
 * grpo_gspo_loss_fwd_bwd — GSPO's sequence-level loss and its dlogits over the kept rollouts.
 * GSPO (Group Sequence Policy Optimization) is one of the base algorithms FastRL is combined with
 * (Sec. 1, Sec. 4); its objective over the kept sequences, with sequence k owning rows
 * [seq_row_off[k], seq_row_off[k+1]) (L_k rows) and advantage A = adv[seq_rollout[k]]:
 *   log s_k = (1/L_k) sum_{t in k} (logp_t - old_logp_t)        (length-normalised ratio)
 *   l_k = -( min(s_k*A, clip(s_k, 1-eps_low, 1+eps_high)*A) - beta*(1/L_k)*sum_t kl_t )
 *   loss = (1/n_seq) sum_k l_k,  kl_t = exp(x_t) - x_t - 1,  x_t = ref_logp_t - logp_t
 *   dlogits[t, v] = w_t*g_t*([v == y] - softmax(z)_v),  w_t = 1/(n_seq*L_k),
 *   g_t = -(c_k*s_k*A + beta*(exp(x_t) - 1)),  c_k = [A>=0][s_k<=1+eps_high] + [A<0][s_k>=1-eps_low]
 * Rows: row t < n_rows reads logits row src = row_index[t] (or t) and y, old_logp, ref_logp at
 *   src, as grpo_loss_fwd_bwd.  Sequences: seq_row_off device i64 [n_seq_rows+1] and
 *   seq_rollout device i32 [n_seq_rows], for instance grpo_compact's kept_off and kept_idx
 *   (n_seq_rows = K, n_rows = T_kept).  Offsets are clamped to [0, n_rows]; rows outside every
 *   sequence get zero gradient.  n_seq > 0: the mean's denominator (the global kept-sequence
 *   count under data parallelism).
 * A sequence with a non-finite log-probability (a token id outside [0, V), non-finite logits)
 *   has no ratio: seq_ratio NaN, no loss term, zero dlogits; the status word says why.
 * Outputs: dlogits [n_rows, V] (dtype dlogits_dtype), logp_out f32 [n_rows] (required),
 *   seq_ratio_out f32 [n_seq_rows] (nullable), loss_out f64 [1], reduced in a fixed order.
 * Workspace: 20 bytes per row + 8 per sequence (size query as everywhere).  Three passes over
 *   the logits' bytes (two reads, one write): log-probabilities with softmax statistics, the
 *   sequence ratios, then dlogits.  Deterministic for a given input.
 * Alignment: as grpo_loss_fwd_bwd; rows that do not start on a 16-byte boundary are realigned,
 *   with the same bits as an aligned call (about 4.2 TB/s against 6.2 at V = 50257 / 50264).
 */
grpo_status grpo_gspo_loss_fwd_bwd(const void* logits, int32_t logits_dtype, int64_t row_stride,
                                   const int64_t* row_index, int64_t n_rows, int32_t V,
                                   const int32_t* y, const float* old_logp, const float* ref_logp,
                                   const float* adv, const int32_t* seq_rollout,
                                   const int64_t* seq_row_off, int32_t n_seq_rows, int64_t n_seq,
                                   float eps_low, float eps_high, float beta, void* dlogits,
                                   int32_t dlogits_dtype, float* logp_out, float* seq_ratio_out,
                                   double* loss_out, int32_t* status, void* ws, size_t* ws_bytes,
                                   grpo_stream_t stream);

/*
 * grpo_gspo_loss_fwd_bwd_dev — grpo_gspo_loss_fwd_bwd with the row and sequence counts read on the
 * device, so that a step with GSPO's loss can be captured in a CUDA graph (as
 * grpo_loss_fwd_bwd_dev for the token-level loss).
 * counts    device i64 [2] = {K, T_kept}, e.g. grpo_compact's counts.  Rows processed:
 *           min(max_rows, T_kept); sequences: min(max_seqs, K); n_seq <= 0 takes K as the mean's
 *           denominator.
 * max_rows, max_seqs  host capacities: dlogits [max_rows, V], logp_out, seq_row_off
 *           [max_seqs+1], seq_rollout, seq_ratio_out and the workspace are sized for them.
 * Entries past the device counts are not written.  All other arguments as
 * grpo_gspo_loss_fwd_bwd.
 */
grpo_status grpo_gspo_loss_fwd_bwd_dev(const void* logits, int32_t logits_dtype,
                                       int64_t row_stride, const int64_t* row_index,
                                       int64_t max_rows, int32_t max_seqs, const int64_t* counts,
                                       int32_t V, const int32_t* y, const float* old_logp,
                                       const float* ref_logp, const float* adv,
                                       const int32_t* seq_rollout, const int64_t* seq_row_off,
                                       int64_t n_seq, float eps_low, float eps_high, float beta,
                                       void* dlogits, int32_t dlogits_dtype, float* logp_out,
                                       float* seq_ratio_out, double* loss_out, int32_t* status,
                                       void* ws, size_t* ws_bytes, grpo_stream_t stream);

/*
 * grpo_lmhead_loss_fwd_bwd — the policy's output layer fused with the GRPO token loss.  Sec. 3.2
 * runs the kept trajectories through the policy, whose last layer maps each token's hidden state
 * to logits over the vocabulary; Eqs. 1-3 give the loss.  Here the logits
 *   z[t, v] = sum_d hidden[t, d] * weight[v, d]
 * are produced on the tensor cores 128 x 256 at a time, one chunk of rows at a time (never all
 * rows at once):
 *   loss, logp_out, row_loss_out: as grpo_loss_fwd_bwd on z (rows in order, row_index = NULL);
 *   dhidden[t, :] = sum_v dlogits[t, v] * weight[v, :]         (chain rule through z = h W^T)
 *   dweight[v, :] = sum_t dlogits[t, v] * hidden[t, :]          (+ the old dweight with
 *                                                                accumulate_dweight != 0)
 * with dlogits = w_t*g_t*([v == y] - softmax(z)_v) rounded to bf16 before the two products.
 * hidden: device bf16, row stride hidden_stride elements (>= D, multiple of 8), 16-byte aligned.
 *   Row t < n_rows reads hidden row src = row_index[t] (device i64, nullable: src = t) and
 *   y[src], old_logp[src], ref_logp[src], as grpo_loss_fwd_bwd reads logits rows; gathered rows
 *   are first copied into the workspace (n_rows * D * 2 bytes).  Outputs are in row order t.
 * weight: device bf16 [V, D], dense, 16-byte aligned.  D: a multiple of 8.
 * adv, row_rollout (indexed by t), eps_low, eps_high, beta, agg_mode, denom_tokens, seq_off,
 *   n_seq, status: as grpo_loss_fwd_bwd.
 * dhidden: device [n_rows, D] (dense), bf16 or f32 per dhidden_dtype.  dweight: device f32
 *   [V, D], overwritten, or added to when accumulate_dweight != 0.
 * dlogits_out: nullable device bf16 [n_rows, grpo_lmhead_dlogits_stride(V)], 16-byte aligned;
 *   when given it receives every row's dlogits (columns >= V are 0) and no chunk buffer is used.
 * logp_out (f32 [n_rows]) and row_loss_out (f64 [n_rows]): nullable.  loss_out: device f64 [1].
 * chunk_rows: rows of logits and dlogits held at a time (rounded up to a multiple of 128); 0
 *   splits the rows into as few equal chunks as keep each chunk's bf16 dlogits within about
 *   4 GiB (their f32 logits then take about 8 GiB).
 *   Smaller chunks need less workspace.
 * Workspace: per row 8 bytes per 256 vocabulary entries of softmax statistics; per chunk row
 *   4 * grpo_lmhead_dlogits_stride(V) bytes of f32 logits (none when grpo_lmhead_tune selects
 *   recomputation) and 2 * grpo_lmhead_dlogits_stride(V) of dlogits (none with dlogits_out); the
 *   f32 partial products of a split K (see grpo_lmhead_grad).
 * Kernels, per chunk: pass 1 (softmax statistics; the chunk's f32 logits stored) and the two
 *   products (grpo_lmhead_grad's) are tcgen05 kernels with TMA operand loads and TMEM
 *   accumulators, one CTA per SM; a row kernel applies Eqs. 1-3 and a streaming kernel forms
 *   dlogits from the stored logits.  The forward results (logp, loss, row terms) do not depend
 *   on chunk_rows or on the launch settings.  Limits: n_rows < 2^31; V >= 1; D >= 8.
 *   Errors: GRPO_ERR_INVALID_ARG for bad sizes, alignment, NULL required pointers;
 *   GRPO_ERR_CUDA when a launch or the tensor-map encoder fails.
 */
grpo_status grpo_lmhead_loss_fwd_bwd(const void* hidden, int64_t hidden_stride,
                                     const int64_t* row_index, int64_t n_rows, const void* weight,
                                     int32_t V, int32_t D, const int32_t* y,
                                     const float* old_logp, const float* ref_logp,
                                     const float* adv, const int32_t* row_rollout, float eps_low,
                                     float eps_high, float beta, int32_t agg_mode,
                                     int64_t denom_tokens, const int64_t* seq_off, int64_t n_seq,
                                     void* dhidden, int32_t dhidden_dtype, float* dweight,
                                     int32_t accumulate_dweight, void* dlogits_out,
                                     float* logp_out, double* row_loss_out, double* loss_out,
                                     int32_t* status, int64_t chunk_rows, void* ws,
                                     size_t* ws_bytes, grpo_stream_t stream);

/*
 * grpo_lmhead_grad — the chain rule through the output layer z = hidden * weight^T for given
 * dlogits (Sec. 3.2: the kept trajectories' hidden states -> logits -> Eqs. 1-3), for instance
 * the bf16 dlogits grpo_loss_fwd_bwd wrote for the kept rows:
 *   dhidden[t, :] = sum_v dlogits[t, v] * weight[v, :]
 *   dweight[v, :] = sum_t dlogits[t, v] * hidden[t, :]   (+ the old dweight with accumulate_dweight)
 * These are the two products grpo_lmhead_loss_fwd_bwd runs after its dlogits pass, on the same
 * tcgen05 kernel: bf16 operands staged by TMA, f32 accumulation in tensor memory, each output
 * rounded once (bf16 dhidden to nearest even).
 * dlogits: device bf16 [n_rows, V] with row stride dlogits_stride (>= V, a multiple of 8).
 * hidden:  device bf16 [n_rows, D] with row stride hidden_stride (>= D, a multiple of 8).
 * weight:  device bf16 [V, D], dense.  D: a positive multiple of 8.  dlogits, hidden and weight
 *   16-byte aligned.
 * dhidden: device [n_rows, D] dense, bf16 or f32 per dhidden_dtype, aligned to its element;
 *   NULL skips it (weight may then be NULL).  dweight: device f32 [V, D]; NULL skips it (hidden
 *   may then be NULL).  n_rows = 0: dweight is zeroed (or left as is when accumulated).
 * status: device i32, nullable (GRPO_DEVFLAG_TIMEOUT if a bounded wait ran out).
 * Workspace: f32 partial products when a product's K is split for load balance (the size query
 *   as everywhere; it may be 0).  Deterministic for a given input and device.
 * Errors: GRPO_ERR_INVALID_ARG for bad sizes, strides, alignment or NULL required pointers;
 *   GRPO_ERR_CUDA when a launch or the tensor-map encoder fails.
 */
grpo_status grpo_lmhead_grad(const void* dlogits, int64_t dlogits_stride, int64_t n_rows,
                             int32_t V, const void* hidden, int64_t hidden_stride,
                             const void* weight, int32_t D, void* dhidden, int32_t dhidden_dtype,
                             float* dweight, int32_t accumulate_dweight, int32_t* status, void* ws,
                             size_t* ws_bytes, grpo_stream_t stream);

/*
 * grpo_lmhead_logp_fwd — log-probability of the sampled token from hidden states, for the old- and
 * reference-policy evaluations of the kept trajectories (Sec. 3.2) through their output layers:
 *   logp_out[t] = z_y - log sum_v exp(z_v),  z = hidden[src] * weight^T,  y = y[src]
 * The pass-1 kernel of grpo_lmhead_loss_fwd_bwd alone (plus its row kernel): no loss, no gradient.
 * hidden, hidden_stride, row_index, n_rows, weight, V, D, y, status: as grpo_lmhead_loss_fwd_bwd.
 * logp_out: device f32 [n_rows] (NaN for a token id outside [0, V)); the same bits as
 * grpo_lmhead_loss_fwd_bwd's logp_out for the same rows.  Workspace: per row 8 bytes per 256
 * vocabulary entries and 4 bytes, plus the gathered rows with row_index.  Limits and errors: as
 * grpo_lmhead_loss_fwd_bwd.
 */
grpo_status grpo_lmhead_logp_fwd(const void* hidden, int64_t hidden_stride,
                                 const int64_t* row_index, int64_t n_rows, const void* weight,
                                 int32_t V, int32_t D, const int32_t* y, float* logp_out,
                                 int32_t* status, void* ws, size_t* ws_bytes, grpo_stream_t stream);

/*
 * grpo_lmhead_gspo_loss_fwd_bwd — the output layer fused with GSPO's sequence-level loss (FastRL on
 * GSPO, Sec. 1, Sec. 4): the objective of grpo_gspo_loss_fwd_bwd on z = hidden * weight^T, with
 * dhidden and dweight by the chain rule as in grpo_lmhead_loss_fwd_bwd.
 * hidden, hidden_stride, row_index, n_rows, weight, V, D, y, old_logp, ref_logp, dhidden,
 *   dhidden_dtype, dweight, accumulate_dweight, dlogits_out, status, chunk_rows: as
 *   grpo_lmhead_loss_fwd_bwd.
 * Sequences: seq_row_off device i64 [n_seq_rows+1] (row offsets in row order t, clamped to
 *   [0, n_rows]) and seq_rollout device i32 [n_seq_rows] (indices into adv), for instance
 *   grpo_compact's kept_off and kept_idx; the loss is the mean over n_seq > 0 sequences.
 * logp_out: device f32 [n_rows], required.  seq_ratio_out: nullable f32 [n_seq_rows] (NaN for a
 *   sequence with an invalid token or no rows).  loss_out: device f64 [1].
 * With no rows or no sequences the loss is 0 and dhidden (and dweight unless accumulated) are 0.
 * Kernels: pass 1 over every row (keeping the first chunk's f32 logits), a row kernel (logp and
 *   softmax statistics), one warp per sequence (ratio, clip, loss term, row gradient scalars),
 *   the fixed-order sum, then per chunk the dlogits and the two GEMMs.  A sequence may cross a
 *   chunk boundary, so no row's dlogits exist before pass 1 has covered every row: the first
 *   chunk's come from its kept logits, each later chunk's from pass 2, which recomputes the
 *   tiles on the tensor cores (every chunk with grpo_lmhead_tune's recompute_logits).  The same
 *   bits either way.
 * Workspace: as grpo_lmhead_loss_fwd_bwd, with 16 bytes per row and 8 per sequence in place of
 *   the per-row loss terms.  Limits and errors: as grpo_lmhead_loss_fwd_bwd.
 */
grpo_status grpo_lmhead_gspo_loss_fwd_bwd(
    const void* hidden, int64_t hidden_stride, const int64_t* row_index, int64_t n_rows,
    const void* weight, int32_t V, int32_t D, const int32_t* y, const float* old_logp,
    const float* ref_logp, const float* adv, const int32_t* seq_rollout,
    const int64_t* seq_row_off, int32_t n_seq_rows, int64_t n_seq, float eps_low, float eps_high,
    float beta, void* dhidden, int32_t dhidden_dtype, float* dweight, int32_t accumulate_dweight,
    void* dlogits_out, float* logp_out, float* seq_ratio_out, double* loss_out, int32_t* status,
    int64_t chunk_rows, void* ws, size_t* ws_bytes, grpo_stream_t stream);

/*
 * grpo_lmhead_tune — launch settings of the output-layer kernels for this process (no counterpart
 * in the paper).  prefetch: k-blocks (64 of D) by which an L2 prefetch of each operand tile runs
 * ahead of its load, 0..64 (0: none).  row_lanes: pairs of 128-row blocks the grid works on at
 * once, 1..8, or 0 to let the library choose per launch.  recompute_logits: 0 (default) lets
 * grpo_lmhead_loss_fwd_bwd store each chunk's f32 logits in pass 1 and form dlogits from them
 * (grpo_lmhead_gspo_loss_fwd_bwd: the first chunk's); 1 makes both recompute the logits in a
 * second tensor-core pass instead (a quarter more FLOPs, 4 bytes per chunk entry less
 * workspace).  The results are the same bits either way.  A size query and the call it sizes
 * must see the same setting.  Returns GRPO_ERR_INVALID_ARG for other values.
 */
grpo_status grpo_lmhead_tune(int32_t prefetch, int32_t row_lanes, int32_t recompute_logits);

/* Row stride, in elements, of grpo_lmhead_loss_fwd_bwd's dlogits_out: V rounded up to a multiple
 * of 32 (0 for V < 1). */
int64_t grpo_lmhead_dlogits_stride(int32_t V);

/*
 * grpo_sum_f64 — *out = v[0] + ... + v[n-1] in fp64, in the same fixed order grpo_loss_fwd_bwd
 * uses for loss_out (bitwise reproducible).  With row_loss_out, a loss computed over rows in
 * several calls (for example chunks of kept rows sharing one dlogits buffer) then sums to
 * exactly the value a single call over all rows gives.
 * v device f64 [n]; out device f64 [1].
 */
grpo_status grpo_sum_f64(const double* v, int64_t n, double* out, grpo_stream_t stream);

/*
 * grpo_loss_fwd_bwd_dev — grpo_loss_fwd_bwd with the row count read on the device, so that a
 * whole step (advantage, prune, compact, loss) is enqueued without a host round trip and can be
 * captured once in a CUDA graph (same Eqs. 1-3).
 * counts    device i64 [2] = {K, T_kept}, e.g. grpo_compact's counts.  Rows processed:
 *           min(max_rows, T_kept).  denom_tokens <= 0 (token mean) takes T_kept as the
 *           denominator and n_seq <= 0 (sequence mean) takes K.
 * max_rows  host capacity: row_index, row_rollout, dlogits [max_rows, V], logp_out and the
 *           workspace (or row_loss_out) are sized for it.
 * All other arguments as grpo_loss_fwd_bwd.
 */
grpo_status grpo_loss_fwd_bwd_dev(const void* logits, int32_t logits_dtype, int64_t row_stride,
                                  const int64_t* row_index, int64_t max_rows, const int64_t* counts,
                                  int32_t V, const int32_t* y, const float* old_logp,
                                  const float* ref_logp, const float* adv,
                                  const int32_t* row_rollout, float eps_low, float eps_high,
                                  float beta, int32_t agg_mode, int64_t denom_tokens,
                                  const int64_t* seq_off, int64_t n_seq, void* dlogits,
                                  int32_t dlogits_dtype, float* logp_out, double* row_loss_out,
                                  double* loss_out, int32_t* status, void* ws, size_t* ws_bytes,
                                  grpo_stream_t stream);

/*
 * grpo_loss_fwd_bwd_noalloc — grpo_loss_fwd_bwd for callers that cannot allocate device memory.
 * The paper has no counterpart: this is an interface convenience of this library.
 * Some callers run the loss where no allocation is possible: a plugin or custom-op host that
 * passes only input and output buffers and has no workspace hook, or a runtime that forbids
 * allocation after start-up to keep its memory footprint fixed.  This entry takes the same
 * arguments as grpo_loss_fwd_bwd without ws/ws_bytes and computes the same results.  Its
 * per-row loss scratch is a fixed array inside the library (2 MiB of fp64, 262144 rows), which
 * every GPU that loads the library holds until the process exits.
 *   - n_rows above 262144 with row_loss_out == NULL returns GRPO_ERR_UNSUPPORTED (pass
 *     row_loss_out, which needs no scratch, or split the rows into several calls).
 *   - The first call on each device looks up the array's device address (cudaGetSymbolAddress)
 *     with that device current, and keeps it for the life of the process.  Under lazy module
 *     loading (the CUDA default) that lookup may also make the driver load this library's GPU
 *     code, array included, which allocates device memory.  So a caller that must not allocate
 *     after start-up makes one call on each device during its start-up phase, before any stream
 *     capture; a call with n_rows = 0 and row_loss_out == NULL is enough (it sets loss_out to 0).
 *   - A device reset (cudaDeviceReset) unloads the array and invalidates the kept address; this
 *     entry must not be called on a device after it has been reset in the same process.
 *   - Every call uses the same array, which keeps the previous call's contents; each call
 *     writes every entry it later reads, so nothing needs clearing.  Calls whose GPU work
 *     overlaps (for instance on two streams at once) race on the array: order them on one
 *     stream.
 *   - It calls no cudaMalloc, cudaFree or other allocating routine.
 */
grpo_status grpo_loss_fwd_bwd_noalloc(const void* logits, int32_t logits_dtype,
                                      int64_t row_stride, const int64_t* row_index,
                                      int64_t n_rows, int32_t V, const int32_t* y,
                                      const float* old_logp, const float* ref_logp,
                                      const float* adv, const int32_t* row_rollout, float eps_low,
                                      float eps_high, float beta, int32_t agg_mode,
                                      int64_t denom_tokens, const int64_t* seq_off, int64_t n_seq,
                                      void* dlogits, int32_t dlogits_dtype, float* logp_out,
                                      double* row_loss_out, double* loss_out, int32_t* status,
                                      grpo_stream_t stream);

/*
 * grpo_loss_tune — launch shape of grpo_loss_fwd_bwd's main kernel for this process.
 * cluster_ctas: CTAs sharing one logits row (1..16, 0 = automatic); threads: 128/256/512
 * (0 = automatic); chunks: copies each CTA splits its slice into (1..16, 0 = automatic).
 * Every shape meets the same accuracy; the shape sets the order of the floating-point sums, so
 * results may differ between shapes in the last bits, and one shape always gives the same bits.
 * grpo_logp_fwd does not use these settings.  Returns GRPO_ERR_INVALID_ARG for other values.
 */
grpo_status grpo_loss_tune(int32_t cluster_ctas, int32_t threads, int32_t chunks);

/*
 * grpo_test_skip_copy — test hook for the bounded-wait path (no counterpart in the paper).
 * With enable != 0, the next grpo_loss_fwd_bwd / grpo_loss_fwd_bwd_dev launch arms the first
 * copy of its first row in one CTA but never issues it.  That CTA's wait runs out after about
 * one second: the kernel ORs GRPO_DEVFLAG_TIMEOUT into the status word and returns normally
 * (that launch's results are invalid); the context stays usable.  Not for production use.
 */
grpo_status grpo_test_skip_copy(int32_t enable);

/*
 * grpo_test_fail_launch — test hook for the error path of every call (no counterpart in the
 * paper).  nth > 0: the nth launch check from now (counting every kernel launch of every call)
 * reports GRPO_ERR_CUDA with an "injected launch failure" message, as a real launch error would;
 * the kernel itself has been enqueued normally, and the call returns without enqueuing the rest.
 * nth = 0 disarms.  Nothing is done to the device.  GRPO_ERR_INVALID_ARG for nth < 0.
 */
grpo_status grpo_test_fail_launch(int32_t nth);

/*
 * Adaptive rollout sampling state, Algorithm 1 (the "adaptive sampling state" and the two
 * epoch-level buffers).  Plain data: it may be copied or saved and restored byte for byte.
 */
typedef struct grpo_ars_state {
  int32_t G1;          /* initial rollout count G_1 */
  int32_t n;           /* rollout count chosen for the next step */
  int32_t have_ref;    /* G'_ref is set */
  int32_t have_gt;     /* G'_t is set */
  double g_ref;        /* G'_ref, Eq. 12 */
  double g_t;          /* G'_t, Eq. 11 */
  double buf_mean_sum; /* sum of the per-step G'^mean values buffered this epoch */
  double buf_max_sum;  /* sum of the per-step G'^max values buffered this epoch */
  int64_t buf_count;   /* number of buffered steps */
} grpo_ars_state;

/* Reset `st` for initial rollout count G1 >= 2 (n = G1, nothing buffered, no reference). */
grpo_status grpo_ars_init(grpo_ars_state* st, int32_t G1);

/*
 * grpo_ars_serialize / grpo_ars_deserialize — checkpoint and resume of the ARS state (no
 * counterpart in the paper, which restarts nothing): a training run that stops mid-epoch resumes
 * with the same buffered means, G'_ref and G'_t, so the rollout counts continue as if
 * uninterrupted.  The record is 64 bytes, little-endian on every host: the tag "FRLARS01", then
 * G1, n, have_ref, have_gt (4 bytes each), g_ref, g_t, buf_mean_sum, buf_max_sum (binary64) and
 * buf_count (8 bytes).
 * serialize: buf == NULL writes the size (64) to *bytes; otherwise *bytes >= 64 is required
 *   (GRPO_ERR_WORKSPACE if smaller) and receives 64.
 * deserialize: GRPO_ERR_INVALID_ARG (st untouched) for a short buffer, a wrong tag, or a state
 *   that grpo_ars_init / adaptive_rollout_count cannot produce (G1 < 2, n outside [2, G1], flags
 *   other than 0 / 1, a negative count, non-finite or negative sums).  Host only.
 */
grpo_status grpo_ars_serialize(const grpo_ars_state* st, void* buf, size_t* bytes);
grpo_status grpo_ars_deserialize(grpo_ars_state* st, const void* buf, size_t bytes);

/*
 * adaptive_rollout_count — ARS update after one step, Eqs. 10-14 and Algorithm 1 (Phases 1a/1b).
 * kept_per_prompt  host i32 [P], P >= 1: |S(q)| of this step.  Their mean and max are buffered
 *                  (Eq. 10).  At an epoch end (epoch_end != 0), with alpha = step/total_steps,
 *                  G'_t = alpha*mean(B_mean) + (1-alpha)*mean(B_max) (Eq. 11); the first epoch end
 *                  also sets G'_ref = (mean(B_mean) + mean(B_max))/2 (Eq. 12); buffers reset.
 * Returns the rollout count for step+1:
 *   max(round(min(G1 - (G'_ref - G'_t), G1)), 2) when both are set and G'_t < G'_ref, else G1
 *   (Eqs. 13-14; round() is round-half-to-even), or -(grpo_status) on an argument error.
 * step is 1-based, 1 <= step <= total_steps.  Host only; touches no GPU.
 */
int32_t adaptive_rollout_count(grpo_ars_state* st, const int32_t* kept_per_prompt, int32_t P,
                               int64_t step, int64_t total_steps, int32_t epoch_end);

#ifdef __cplusplus
}
#endif

#endif /* FASTRL_GRPO_H_ */
