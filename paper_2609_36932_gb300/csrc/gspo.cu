// grpo_gspo_loss_fwd_bwd: GSPO's sequence-level loss and its dlogits over the kept rollouts.
// GSPO (Group Sequence Policy Optimization, Zheng et al., 2025) is one of the base algorithms
// FastRL is combined with (Sec. 1, Sec. 4): the importance ratio is taken per sequence,
//   log s_k = (1/L_k) sum_{t in k} (logp_t - old_logp_t),
// and clipped per sequence.  A token's gradient therefore depends on every log-probability of its
// sequence, so one fused pass over the logits cannot produce it.  Three passes:
//   1. the forward-only row kernel (loss.cu) writes logp and each row's softmax statistics
//      {M, S = sum exp(z - M), S without y}: one read of the logits;
//   2. gspo_seq_kernel, one warp per sequence: s_k, the clip decision, the sequence's loss term
//      and every row's gradient coefficient w_t * g_t (a few bytes per row);
//   3. gspo_dlogits_kernel streams the logits once more and writes
//      dlogits = coef * ([v == y] - exp(z - M) / S), with pass B's arithmetic from loss.cu.
// Traffic per kept row: 2 reads and 1 write of V entries (vs 1 + 1 for the token-level loss).
#define GRPO_TU 4  // this file's bit in the checked build's report (grpo_debug_checks)
#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "trace.cuh"
#include "rowops.cuh"

namespace fastrl {
namespace {

struct SeqArgs {
  const float* logp;
  const int64_t* row_index;
  const float* old_logp;
  const float* ref_logp;
  const float* adv;
  const int32_t* seq_rollout;
  const int64_t* seq_row_off;
  int32_t n_seq_rows;
  int64_t n_rows;
  double lo, hi;  // 1 - eps_low, 1 + eps_high in fp64
  float beta;
  double inv_nseq;
  // device counts {K, T_kept} (nullable): sequences min(n_seq_rows, K), rows min(n_rows, T_kept);
  // with nseq_from_counts the mean's denominator is K
  const int64_t* counts;
  int32_t nseq_from_counts;
  float* coef;
  double* seq_loss;
  float* seq_ratio;
};

constexpr int kSeqWarps = 8;

// One warp per sequence.  Lane-strided fp64 partial sums combined by a fixed xor-shuffle tree:
// the result depends only on the sequence's rows, not on scheduling.
__global__ void __launch_bounds__(kSeqWarps * 32) gspo_seq_kernel(const SeqArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t k = (int64_t)blockIdx.x * kSeqWarps + (threadIdx.x >> 5);
  int64_t n_seqs = a.n_seq_rows, n_rows = a.n_rows;
  double inv_nseq = a.inv_nseq;
  if (a.counts) {
    n_seqs = a.counts[0] < n_seqs ? a.counts[0] : n_seqs;
    n_rows = a.counts[1] < n_rows ? a.counts[1] : n_rows;
    if (a.nseq_from_counts) inv_nseq = a.counts[0] > 0 ? 1.0 / (double)a.counts[0] : 0.0;
  }
  if (k >= n_seqs) return;
  int64_t r0 = a.seq_row_off[k], r1 = a.seq_row_off[k + 1];
  r0 = r0 < 0 ? 0 : (r0 > n_rows ? n_rows : r0);  // offsets outside [0, n_rows] are clamped
  r1 = r1 < r0 ? r0 : (r1 > n_rows ? n_rows : r1);
  const int64_t L = r1 - r0;
  double slr = 0.0, skl = 0.0;
  int bad = 0;
  for (int64_t t = r0 + lane; t < r1; t += 32) {
    int64_t src = a.row_index ? a.row_index[t] : t;
    if (!GRPO_DCHECK(src >= 0)) src = 0;
    const float lp = a.logp[t];
    if (!isfinite(lp)) bad = 1;
    slr += (double)lp - (double)a.old_logp[src];
    const float x = a.ref_logp[src] - lp;
    skl += (double)(expm1f(x) - x);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    slr += __shfl_xor_sync(0xffffffffu, slr, o);
    skl += __shfl_xor_sync(0xffffffffu, skl, o);
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
  }
  if (L == 0 || bad) {  // no ratio: the sequence contributes nothing
    for (int64_t t = r0 + lane; t < r1; t += 32) a.coef[t] = 0.f;
    if (lane == 0) {
      a.seq_loss[k] = 0.0;
      if (a.seq_ratio) a.seq_ratio[k] = __int_as_float(0x7fc00000);
    }
    return;
  }
  int32_t ro = a.seq_rollout[k];
  if (!GRPO_DCHECK(ro >= 0)) ro = 0;
  const double A = (double)a.adv[ro];
  const double s = exp(slr / (double)L);
  const double clipped = fmin(fmax(s, a.lo), a.hi);
  const double surr = fmin(s * A, clipped * A);
  const bool c = (A >= 0.0) ? (s <= a.hi) : (s >= a.lo);
  if (lane == 0) {
    a.seq_loss[k] = -(surr - (double)a.beta * skl / (double)L) * inv_nseq;
    if (a.seq_ratio) a.seq_ratio[k] = (float)s;
  }
  const float w = (float)(inv_nseq / (double)L);
  const float sa = c ? (float)(s * A) : 0.f;
  for (int64_t t = r0 + lane; t < r1; t += 32) {
    int64_t src = a.row_index ? a.row_index[t] : t;
    if (!GRPO_DCHECK(src >= 0)) src = 0;
    const float x = a.ref_logp[src] - a.logp[t];
    a.coef[t] = w * -(sa + a.beta * expm1f(x));
  }
}

struct DlArgs {
  const char* logits;
  int64_t row_stride_bytes;
  const int64_t* row_index;
  int64_t n_rows;
  int32_t V;
  const int32_t* y;
  const float4* stats;
  const float* coef;
  char* dlogits;
  int32_t vec;      // input rows 16-byte aligned: vector loads
  int32_t out_vec;  // output rows 16-byte aligned: vector stores
  int32_t tiles_per_row;
  const int64_t* counts;  // nullable: rows min(n_rows, counts[1])
};

constexpr int kDlThreads = 256;
constexpr int kDlUnroll = 4;  // 16-byte vectors per thread per tile

// Persistent grid over tiles (row, segment of kDlThreads * kDlUnroll vectors).  Each thread
// issues its kDlUnroll loads before using any of them.
// kAny: the instance for rows that need not start on a 16-byte boundary (chosen by the host
// only then).  A segment is kDlThreads * kDlUnroll aligned 16-byte words of the dlogits row;
// each word's inputs come from the aligned words of the logits row that hold them
// (pairs_at_global), and the first and last few elements of the row are stored one by one.
template <typename InT, typename OutT, bool kAny>
__global__ void __launch_bounds__(kDlThreads) gspo_dlogits_kernel(const DlArgs a) {
  constexpr int kVec = Fmt<InT>::kVec;
  constexpr int kPairs = Fmt<InT>::kPairs;
  constexpr int kSeg = kDlThreads * kDlUnroll;
  const int tid = threadIdx.x;
  const float2 l2e2 = make_float2(kLog2e, kLog2e);
  const int nvec = a.vec ? a.V / kVec : 0;
  const int tail0 = nvec * kVec;
  int64_t n_rows = a.n_rows;
  if (a.counts && a.counts[1] < n_rows) n_rows = a.counts[1];
  const int64_t n_tiles = n_rows * a.tiles_per_row;
  for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int64_t row = tile / a.tiles_per_row;
    const int seg = (int)(tile - row * a.tiles_per_row);
    const bool last_seg = seg == a.tiles_per_row - 1;
    OutT* orow = reinterpret_cast<OutT*>(a.dlogits) + row * (int64_t)a.V;
    int64_t src = a.row_index ? a.row_index[row] : row;
    if (!GRPO_DCHECK(src >= 0)) src = 0;
    const InT* grow = reinterpret_cast<const InT*>(a.logits + src * a.row_stride_bytes);
    const float coef = a.coef[row];
    // vector loads and stores need 16-byte aligned rows (the host sets vec / out_vec from that)
    if (!GRPO_DCHECK((!a.vec || (reinterpret_cast<uintptr_t>(grow) & 15u) == 0) &&
                     (!a.out_vec || (reinterpret_cast<uintptr_t>(orow) & 15u) == 0)))
      continue;
    const int j0 = seg * kSeg;
    if constexpr (kAny) {
      using OW = OutWord<InT, OutT>;
      constexpr int E = OW::kElems;
      const int omis = (int)(reinterpret_cast<uintptr_t>(orow) & 15u);
      const int h = min(a.V, ((16 - omis) & 15) / (int)sizeof(OutT));  // elements before word 0
      const int nfull = (a.V - h) / E;
      const int rest0 = h + nfull * E;
      float neg_scale = 0.f, dy = 0.f, shB = 0.f;
      int32_t yv = -1;
      if (coef != 0.f) {
        const float4 st = a.stats[row];  // {M, S, S without y}
        yv = a.y[src];
        neg_scale = -coef / st.y;
        dy = coef * (st.z / st.y);
        shB = -st.x * kLog2e;
        if (fabsf(neg_scale) >= 0x1p-100f) {
          shB += kShiftB;
          neg_scale *= 0x1p-16f;
        }
      }
      const float2 shb2 = make_float2(shB, shB), ns2 = make_float2(neg_scale, neg_scale);
      float2 p[kDlUnroll][OW::kPairs];
#pragma unroll
      for (int u = 0; u < kDlUnroll; ++u) {
        const int w = j0 + u * kDlThreads + tid;
        if (coef != 0.f && w < nfull) pairs_at_global<InT, OutT>(grow, a.V, h + w * E, p[u]);
      }
#pragma unroll
      for (int u = 0; u < kDlUnroll; ++u) {
        const int w = j0 + u * kDlThreads + tid;
        if (w >= nfull) continue;
        const int i0 = h + w * E;
        float2 d[OW::kPairs];
#pragma unroll
        for (int i = 0; i < OW::kPairs; ++i)
          d[i] = coef != 0.f ? __fmul2_rn(ex2x2(__ffma2_rn(p[u][i], l2e2, shb2)), ns2)
                             : make_float2(0.f, 0.f);
        const int yi = yv - i0;
        if (coef != 0.f && (unsigned)yi < (unsigned)E) {
#pragma unroll
          for (int i = 0; i < OW::kPairs; ++i) {
            if (2 * i == yi) d[i].x = dy;
            if (2 * i + 1 == yi) d[i].y = dy;
          }
        }
        store_pairs<OutT, OW::kPairs>(orow + i0, d);
      }
      if (last_seg) {
        for (int t = tid; t < h + (a.V - rest0); t += kDlThreads) {
          const int e = t < h ? t : rest0 + (t - h);  // the head, then the tail
          float d = 0.f;
          if (coef != 0.f) {
            d = neg_scale * ex2(fmaf(Fmt<InT>::load(grow + e), kLog2e, shB));
            if (e == yv) d = dy;
          }
          Fmt<OutT>::store(orow + e, d);
        }
      }
      continue;
    }
    if (coef == 0.f) {  // clipped, zero-advantage without KL, or no ratio: a zero row
      float2 d[kPairs];
#pragma unroll
      for (int i = 0; i < kPairs; ++i) d[i] = make_float2(0.f, 0.f);
      for (int u = 0; u < kDlUnroll; ++u) {
        const int j = j0 + u * kDlThreads + tid;
        if (j < nvec) {
          if (a.out_vec)
            store_pairs<OutT, kPairs>(orow + j * kVec, d);
          else
            store_pairs_scalar<OutT, kPairs>(orow + j * kVec, d);
        }
      }
      if (last_seg)
        for (int e = tail0 + tid; e < a.V; e += kDlThreads) Fmt<OutT>::store(orow + e, 0.f);
      continue;
    }
    const float4 st = a.stats[row];  // {M, S, S without y}
    const int32_t yv = a.y[src];
    float neg_scale = -coef / st.y;
    const float dy = coef * (st.z / st.y);
    float shB = -st.x * kLog2e;
    if (fabsf(neg_scale) >= 0x1p-100f) {  // as pass B of the fused loss (kShiftB)
      shB += kShiftB;
      neg_scale *= 0x1p-16f;
    }
    const float2 shb2 = make_float2(shB, shB), ns2 = make_float2(neg_scale, neg_scale);
    uint4 q[kDlUnroll];
#pragma unroll
    for (int u = 0; u < kDlUnroll; ++u) {
      const int j = j0 + u * kDlThreads + tid;
      if (j < nvec) q[u] = __ldcs(reinterpret_cast<const uint4*>(grow) + j);
    }
#pragma unroll
    for (int u = 0; u < kDlUnroll; ++u) {
      const int j = j0 + u * kDlThreads + tid;
      if (j >= nvec) continue;
      float2 p[kPairs], d[kPairs];
      Fmt<InT>::pairs(q[u], p);
#pragma unroll
      for (int i = 0; i < kPairs; ++i) d[i] = __fmul2_rn(ex2x2(__ffma2_rn(p[i], l2e2, shb2)), ns2);
      const int yi = yv - j * kVec;
      if ((unsigned)yi < (unsigned)kVec) {
#pragma unroll
        for (int i = 0; i < kPairs; ++i) {
          if (2 * i == yi) d[i].x = dy;
          if (2 * i + 1 == yi) d[i].y = dy;
        }
      }
      if (a.out_vec)
        store_pairs<OutT, kPairs>(orow + j * kVec, d);
      else
        store_pairs_scalar<OutT, kPairs>(orow + j * kVec, d);
    }
    if (last_seg) {
      for (int e = tail0 + tid; e < a.V; e += kDlThreads) {
        float d = neg_scale * ex2(fmaf(Fmt<InT>::load(grow + e), kLog2e, shB));
        if (e == yv) d = dy;
        Fmt<OutT>::store(orow + e, d);
      }
    }
  }
}

using DlKernel = void (*)(DlArgs);

template <bool kAny>
DlKernel dl_kernel_of(int in_dtype, int out_dtype) {
  if (in_dtype == GRPO_DTYPE_BF16)
    return out_dtype == GRPO_DTYPE_BF16 ? gspo_dlogits_kernel<__nv_bfloat16, __nv_bfloat16, kAny>
                                        : gspo_dlogits_kernel<__nv_bfloat16, float, kAny>;
  return out_dtype == GRPO_DTYPE_BF16 ? gspo_dlogits_kernel<float, __nv_bfloat16, kAny>
                                      : gspo_dlogits_kernel<float, float, kAny>;
}
DlKernel dl_kernel_for(int in_dtype, int out_dtype, bool any) {
  return any ? dl_kernel_of<true>(in_dtype, out_dtype) : dl_kernel_of<false>(in_dtype, out_dtype);
}

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int g_dl_blocks[kMaxDevices][8] = {};  // resident blocks per SM x SMs, per device and instance

struct GspoWs {
  float4* stats;
  float* coef;
  double* seq_loss;
};

size_t gspo_ws_bytes(int64_t n_rows, int64_t n_seq_rows) {
  return align_up((size_t)n_rows * 16, 256) + align_up((size_t)n_rows * 4, 256) +
         align_up((size_t)n_seq_rows * 8, 256);
}

GspoWs gspo_ws(void* ws, int64_t n_rows) {
  char* p = static_cast<char*>(ws);
  GspoWs w;
  w.stats = reinterpret_cast<float4*>(p);
  p += align_up((size_t)n_rows * 16, 256);
  w.coef = reinterpret_cast<float*>(p);
  p += align_up((size_t)n_rows * 4, 256);
  w.seq_loss = reinterpret_cast<double*>(p);
  return w;
}

}  // namespace
}  // namespace fastrl

using namespace fastrl;

namespace fastrl {
namespace {

// n_rows / n_seq_rows: exact counts, or with counts (device {K, T_kept}) capacities whose used
// part the kernels read on the device; then n_seq <= 0 takes K as the denominator.
grpo_status gspo_impl(const char* who, const void* logits, int32_t logits_dtype, int64_t row_stride,
                      const int64_t* row_index, int64_t n_rows, int32_t V, const int32_t* y,
                      const float* old_logp, const float* ref_logp, const float* adv,
                      const int32_t* seq_rollout, const int64_t* seq_row_off, int32_t n_seq_rows,
                      const int64_t* counts, int64_t n_seq, float eps_low, float eps_high,
                      float beta, void* dlogits, int32_t dlogits_dtype, float* logp_out,
                      float* seq_ratio_out, double* loss_out, int32_t* status, void* ws,
                      size_t* ws_bytes, grpo_stream_t stream) {
  if (logits_dtype != GRPO_DTYPE_BF16 && logits_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: logits_dtype = %d", who, logits_dtype);
  if (dlogits_dtype != GRPO_DTYPE_BF16 && dlogits_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: dlogits_dtype = %d", who, dlogits_dtype);
  if (n_rows < 0 || n_rows >= (int64_t(1) << 31) || n_seq_rows < 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: n_rows = %lld, n_seq_rows = %d", who, (long long)n_rows,
                n_seq_rows);
  if (V < 1 || row_stride < V)
    return fail(GRPO_ERR_INVALID_ARG, "%s: V = %d, row_stride = %lld", who, V, (long long)row_stride);
  if (n_seq <= 0 && counts == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "%s: n_seq = %lld", who, (long long)n_seq);
  if (!(beta >= 0.f) || !(eps_low >= 0.f) || !(eps_high >= 0.f))
    return fail(GRPO_ERR_INVALID_ARG, "%s: beta, eps_low, eps_high must be >= 0", who);
  const size_t need = gspo_ws_bytes(n_rows, n_seq_rows);
  bool query = false;
  grpo_status st = workspace_check(ws, ws_bytes, need, who, &query);
  if (st != GRPO_OK || query) return st;
  if (!loss_out) return fail(GRPO_ERR_INVALID_ARG, "%s: loss_out is NULL", who);
  if (n_seq_rows > 0 && (!seq_row_off || !seq_rollout || !adv))
    return fail(GRPO_ERR_INVALID_ARG, "%s: NULL sequence array", who);
  if (n_rows > 0 && (!logits || !y || !old_logp || !ref_logp || !dlogits || !logp_out))
    return fail(GRPO_ERR_INVALID_ARG, "%s: NULL array", who);
  if (n_rows > 0 && reinterpret_cast<uintptr_t>(dlogits) % (dlogits_dtype == GRPO_DTYPE_BF16 ? 2 : 4))
    return fail(GRPO_ERR_INVALID_ARG, "%s: dlogits not aligned to its element size", who);
  cudaStream_t s = as_stream(stream);
  cudaError_t e = cudaSuccess;
  if (n_seq_rows == 0) {  // no sequences: the loss is 0 and every row's gradient is 0
    if (n_rows > 0) {
      const size_t out_bytes = dlogits_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
      e = cudaMemsetAsync(dlogits, 0, (size_t)n_rows * V * out_bytes, s);
      if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: memset: %s", who, cudaGetErrorString(e));
    }
    return grpo_sum_f64(nullptr, 0, loss_out, stream);
  }
  const GspoWs w = gspo_ws(ws, n_rows);

  // 1. log-probabilities and softmax statistics
  if (n_rows > 0) {
    st = logp_rows(who, logits, logits_dtype, row_stride, row_index, n_rows, counts, V, y,
                   logp_out, w.stats, status, s);
    if (st != GRPO_OK) return st;
    // rows outside every sequence keep coef 0
    e = cudaMemsetAsync(w.coef, 0, (size_t)n_rows * 4, s);
    if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: memset: %s", who, cudaGetErrorString(e));
  }

  // 2. sequence ratios, loss terms, row coefficients
  SeqArgs sa = {};
  sa.logp = logp_out;
  sa.row_index = row_index;
  sa.old_logp = old_logp;
  sa.ref_logp = ref_logp;
  sa.adv = adv;
  sa.seq_rollout = seq_rollout;
  sa.seq_row_off = seq_row_off;
  sa.n_seq_rows = n_seq_rows;
  sa.n_rows = n_rows;
  sa.lo = 1.0 - (double)eps_low;
  sa.hi = 1.0 + (double)eps_high;
  sa.beta = beta;
  sa.inv_nseq = n_seq > 0 ? 1.0 / (double)n_seq : 0.0;
  sa.counts = counts;
  sa.nseq_from_counts = n_seq <= 0 ? 1 : 0;
  sa.coef = w.coef;
  sa.seq_loss = w.seq_loss;
  sa.seq_ratio = seq_ratio_out;
  gspo_seq_kernel<<<(unsigned)((n_seq_rows + kSeqWarps - 1) / kSeqWarps), kSeqWarps * 32, 0, s>>>(sa);
  count_launches(1);
  st = check_launch(who);
  if (st != GRPO_OK) return st;

  // 3. dlogits, streaming
  const int64_t* k_dev = counts ? counts : nullptr;  // the sum runs over min(n_seq_rows, K) terms
  if (n_rows == 0) return launch_sum_rows(w.seq_loss, n_seq_rows, k_dev, loss_out, s, who);
  const int in_bytes = logits_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  const int out_bytes = dlogits_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  const int vec_elems = 16 / in_bytes;
  DlArgs da = {};
  da.logits = static_cast<const char*>(logits);
  da.row_stride_bytes = row_stride * in_bytes;
  da.row_index = row_index;
  da.n_rows = n_rows;
  da.V = V;
  da.y = y;
  da.stats = w.stats;
  da.coef = w.coef;
  da.dlogits = static_cast<char*>(dlogits);
  da.vec = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && (da.row_stride_bytes % 16 == 0);
  da.out_vec = (reinterpret_cast<uintptr_t>(dlogits) % 16 == 0) && (((int64_t)V * out_bytes) % 16 == 0);
  const bool any = !da.vec || !da.out_vec;  // kAny: segments of 16-byte output words
  const int nvec = any ? (V * out_bytes + 15) / 16 : V / vec_elems;
  da.tiles_per_row = std::max(1, (nvec + kDlThreads * kDlUnroll - 1) / (kDlThreads * kDlUnroll));
  da.counts = counts;
  const DlKernel fn = dl_kernel_for(logits_dtype, dlogits_dtype, any);
  const int inst = (logits_dtype == GRPO_DTYPE_BF16 ? 0 : 2) + (dlogits_dtype == GRPO_DTYPE_BF16 ? 0 : 1) +
                   (any ? 4 : 0);
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: cudaGetDevice: %s", who, cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices)
    return fail(GRPO_ERR_UNSUPPORTED, "%s: device %d beyond %d", who, dev, kMaxDevices);
  int resident = 0;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    resident = g_dl_blocks[dev][inst];
    if (resident == 0) {
      int per_sm = 0, sms = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kDlThreads, 0);
      if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "%s: occupancy query: %s", who, cudaGetErrorString(e));
      resident = std::max(1, per_sm) * std::max(1, sms);
      g_dl_blocks[dev][inst] = resident;
    }
  }
  const int64_t n_tiles = n_rows * da.tiles_per_row;
  const unsigned grid = (unsigned)std::min<int64_t>(n_tiles, resident);
  fn<<<grid, kDlThreads, 0, s>>>(da);
  count_launches(1);
  st = check_launch(who);
  if (st != GRPO_OK) return st;

  // 4. the loss: the sequences' terms summed in a fixed order
  return launch_sum_rows(w.seq_loss, n_seq_rows, k_dev, loss_out, s, who);
}

}  // namespace
}  // namespace fastrl

extern "C" grpo_status grpo_gspo_loss_fwd_bwd(
    const void* logits, int32_t logits_dtype, int64_t row_stride, const int64_t* row_index,
    int64_t n_rows, int32_t V, const int32_t* y, const float* old_logp, const float* ref_logp,
    const float* adv, const int32_t* seq_rollout, const int64_t* seq_row_off, int32_t n_seq_rows,
    int64_t n_seq, float eps_low, float eps_high, float beta, void* dlogits, int32_t dlogits_dtype,
    float* logp_out, float* seq_ratio_out, double* loss_out, int32_t* status, void* ws,
    size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_gspo_loss_fwd_bwd");
  clear_error();
  return gspo_impl("grpo_gspo_loss_fwd_bwd", logits, logits_dtype, row_stride, row_index, n_rows,
                   V, y, old_logp, ref_logp, adv, seq_rollout, seq_row_off, n_seq_rows, nullptr,
                   n_seq, eps_low, eps_high, beta, dlogits, dlogits_dtype, logp_out,
                   seq_ratio_out, loss_out, status, ws, ws_bytes, stream);
}

extern "C" grpo_status grpo_gspo_loss_fwd_bwd_dev(
    const void* logits, int32_t logits_dtype, int64_t row_stride, const int64_t* row_index,
    int64_t max_rows, int32_t max_seqs, const int64_t* counts, int32_t V, const int32_t* y,
    const float* old_logp, const float* ref_logp, const float* adv, const int32_t* seq_rollout,
    const int64_t* seq_row_off, int64_t n_seq, float eps_low, float eps_high, float beta,
    void* dlogits, int32_t dlogits_dtype, float* logp_out, float* seq_ratio_out, double* loss_out,
    int32_t* status, void* ws, size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_gspo_loss_fwd_bwd_dev");
  clear_error();
  if (counts == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_gspo_loss_fwd_bwd_dev: counts is NULL");
  return gspo_impl("grpo_gspo_loss_fwd_bwd_dev", logits, logits_dtype, row_stride, row_index,
                   max_rows, V, y, old_logp, ref_logp, adv, seq_rollout, seq_row_off, max_seqs,
                   counts, n_seq, eps_low, eps_high, beta, dlogits, dlogits_dtype, logp_out,
                   seq_ratio_out, loss_out, status, ws, ws_bytes, stream);
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_gspo)
}  // namespace fastrl
