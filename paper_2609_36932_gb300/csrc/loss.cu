// grpo_loss_fwd_bwd: fused GRPO token loss and dlogits, Sec. 3.1 Eqs. 1-3, one read of the
// logits and one write of the gradient; and grpo_logp_fwd, the log-probabilities alone.
//
// Fused loss (HBM-bound: ~2 bytes read + 2-4 bytes written per vocabulary entry, ~10 flops):
//   * A row of V logits is split over a cluster of C CTAs; CTA c holds the slice
//     [c*slice, (c+1)*slice) of the row in shared memory for the whole row, so the logits are
//     read from HBM exactly once.  (V = 152064 bf16 is 297 KiB, more than one SM holds; by
//     default C = 4 with bf16 dlogits, 74 KiB slices and 3 CTAs per SM, and C = 8 with f32.)
//   * Each slice arrives by non-tensor bulk copies (cp.async.bulk, 16-byte granules) in a few
//     chunks, each completing on its own mbarrier, so the CTA starts reducing chunk 0 while
//     the rest is in flight.
//   * Roles: the consumer warps compute; one producer warp (one lane) stages each row's inputs
//     (source row, token and its logit z_y, advantage, old/reference log-probs, weight) in
//     shared memory and issues the slice's copies.  Nothing in the row loop waits for the whole
//     CTA.
//   * Pass A: per-thread online max and sum of exp (base 2, MUFU ex2) over the slice, leaving
//     out the sampled token y; warp shuffles combine a warp's threads.
//   * Exchange: each warp pushes its (max, sum) into every cluster peer's shared memory with
//     st.async, which completes bytes on the peer's mbarrier (no cluster-wide barrier);
//     each warp then waits on its own CTA's mbarrier, combines the C x warps entries and forms
//     the row's log-sum-exp, log-prob, ratio, clipped surrogate, KL term and gradient
//     coefficient itself.  Every warp of the cluster computes the same numbers.
//   * Pass B: dlogits[v] = -coef * exp(z_v - lse) (+coef at v = y) from the shared-memory slice,
//     written with 16-byte streaming stores.  A warp that has finished chunk k arrives on that
//     chunk's release mbarrier; once all have, the producer copies chunk k of the cluster's next
//     row into the same buffer.
//   * The grid is persistent: as many clusters as fit at once; cluster i takes rows i, i+n, ...
//   * Rows that do not start on a 16-byte boundary run the kAny instance (see the kernel).
//   * Per-row loss terms go to a buffer; a fixed-order cluster reduction (reduce.cu) sums them.
// Every wait on a copy is bounded (about one second); on expiry the kernel records
// GRPO_DEVFLAG_TIMEOUT, stops waiting and issuing copies, and runs to the end.
//
// Log-probabilities alone (logp_stream_kernel, also GSPO's first pass): no gradient pass, so no
// slice to keep; one CTA streams each row, and every CTA of the persistent grid is resident.
#define GRPO_TU 3  // this file's bit in the checked build's report (grpo_debug_checks)
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <type_traits>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>

#include "common.cuh"
#include "trace.cuh"
#include "rowops.cuh"

namespace fastrl {
namespace {

constexpr uint64_t kWaitLimitNs = 1000000000ull;
constexpr int kMaxChunks = 16;
constexpr int kMaxCluster = 16;

struct LossArgs {
  const char* logits;
  int64_t row_stride_bytes;
  const int64_t* row_index;
  int64_t n_rows;
  int32_t V;
  const int32_t* y;
  const float* old_logp;
  const float* ref_logp;
  const float* adv;
  const int32_t* row_rollout;
  // Clip bounds 1 - eps_low and 1 + eps_high are defined in fp64.  For an f32 ratio rho,
  // rho <= hi_dn and rho >= lo_up decide exactly as the fp64 comparisons (hi_dn: largest f32
  // <= 1 + eps_high; lo_up: smallest f32 >= 1 - eps_low); clamped values round to nearest.
  // The row scalars then need no fp64 arithmetic, which is scarce on this GPU.
  float lo_up, hi_dn, lo_rn, hi_rn;
  float beta;
  int32_t agg_mode;
  double inv_denom;  // agg 0: 1 / denom_tokens
  float inv_denom_f;
  const int64_t* seq_off;
  float inv_nseq_f;  // agg 1: 1 / n_seq
  char* dlogits;
  float* logp_out;
  float4* stats_out;  // logp_stream_kernel, nullable: per row {max, sum of exp, that sum without y, 0}
  double* row_loss;
  int32_t* status;
  int32_t slice;       // elements per CTA, a multiple of the 16-byte vector width
  int32_t chunk_vecs;  // 16-byte vectors per copy
  int32_t n_chunks;
  int32_t bulk;     // rows 16-byte aligned: slices arrive by bulk copies
  int32_t out_vec;  // dlogits rows 16-byte aligned: vector stores
  // Device counts {K, T_kept} (nullable): rows processed = min(n_rows, T_kept); with
  // denom_from_counts the token-mean denominator is T_kept and Eq. 1's n_seq is K.
  const int64_t* counts;
  int32_t denom_from_counts;
  int32_t skip_copy;  // test hook (grpo_test_skip_copy): one copy is armed but never issued
};

// ---- PTX helpers ------------------------------------------------------------------------------

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
// Test the phase; while it is incomplete the thread may be suspended for up to ~0.1 ms
// (the hint, in ns) instead of spinning and taking issue slots.
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(100000u)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint32_t mapa_shared(uint32_t local_addr, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local_addr), "r"(rank));
  return remote;
}
__device__ __forceinline__ void bulk_copy_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
// Ask L2 to fetch [src, src + bytes) (16-byte aligned, a multiple of 16 bytes); no completion.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}
// Combine two (max, sum of exp relative to max) pairs.
__device__ __forceinline__ void lse_combine(float& m, float& s, float mo, float so) {
  const float M = fmaxf(m, mo);
  const float a = (m == -INFINITY) ? 0.f : s * ex2((m - M) * kLog2e);
  const float b = (mo == -INFINITY) ? 0.f : so * ex2((mo - M) * kLog2e);
  m = M;
  s = a + b;
}

// ---- the kernel -------------------------------------------------------------------------------

// A row's inputs, staged in shared memory by the producer warp (one slot per row parity): the
// logits row, the sampled token, its logit z_y (0 for a token outside [0, V)), the advantage, the
// old and reference log-probabilities and the row's weight.
struct __align__(16) RowIn {
  int64_t src;
  int32_t y;
  float zy, A, old_lp, ref_lp, w;
};
static_assert(sizeof(RowIn) == 32, "row slot");

// Shared memory of one CTA after its slice (sized for the launch's chunk count, so that at the
// default V = 152064 shape three CTAs still fit an SM): copy barriers (full and empty per chunk),
// two exchange barriers, the abort flag (16 bytes), two row slots, then the exchange entries
// [2][C * warps], one (max, sum) pair each.
__host__ __device__ constexpr int loss_smem_fixed(int n_chunks) {
  return (2 * n_chunks + 2) * 8 + 16 + 2 * (int)sizeof(RowIn);
}

// 8-byte store into a cluster peer's shared memory that completes 8 bytes of that peer's
// mbarrier transaction count.
__device__ __forceinline__ void st_async_f2(uint32_t remote_addr, float2 v, uint32_t remote_bar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(
          remote_addr),
      "f"(v.x), "f"(v.y), "r"(remote_bar)
      : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// kCap: compile for 1536 resident threads per SM (1024 when the output is wider than the input),
// the producer warp included.  Used when the slice is small enough that shared memory would allow
// that many threads.  Otherwise the instance is compiled for the CTAs per SM that shared memory
// admits at its default shapes: 3 with 256 consumer threads (V = 152064, bf16 in and out), 7 with
// 128 (V = 32000; V = 152064 with f32 dlogits admits 5).  Without that bound the compiler settled
// at 56 registers with a small spill; with a bound of 1 it took 88, one CTA per SM fewer.
template <typename InT, typename OutT>
constexpr int kResidentThreads = sizeof(OutT) > sizeof(InT) ? 1024 : 1536;
constexpr int uncapped_ctas(int threads) { return threads == 256 ? 3 : (threads == 128 ? 7 : 1); }
template <typename InT, typename OutT, int kThreads, bool kCap>
constexpr int kMinCtas = kCap ? kResidentThreads<InT, OutT> / (kThreads + 32) : uncapped_ctas(kThreads);

// kThreads consumer threads (kThreads / 32 warps) and one producer warp.  No CTA-wide barrier
// inside the row loop: the producer refills chunk k of the next row as soon as every consumer
// warp has released it (an mbarrier per chunk), and each consumer warp exchanges its own partial
// (max, sum) with the cluster and forms the row's scalars itself.
//
// kAny: the instance for rows that need not start on a 16-byte boundary (an odd V stored
// densely, a row stride that is not a multiple of 16 bytes, an unaligned base), chosen by the
// host only for such launches.  Per row and slice: an aligned slice still arrives by bulk
// copies; an unaligned one is realigned by the consumers, each 16-byte vector assembled from
// the two aligned words that hold it (extract16), except a vector whose words would reach
// outside the row, which is loaded element by element.  A dlogits row that does not start on a
// 16-byte boundary is written as aligned 16-byte words read at an offset from the shared-memory
// slice (pairs_at), with the slice's first and last few elements stored one by one.  The
// consumers pass a named barrier between pass A and pass B, since those reads cross vectors
// that other threads wrote.
template <typename InT, typename OutT, int kThreads, bool kCap, bool kAny>
__global__ void __launch_bounds__(kThreads + 32, (kMinCtas<InT, OutT, kThreads, kCap>))
    grpo_loss_kernel(const LossArgs a) {
  constexpr int kVec = Fmt<InT>::kVec;
  constexpr int kPairs = Fmt<InT>::kPairs;
  constexpr int kWarps = kThreads / 32;  // consumer warps; warp kWarps is the producer
  // Two vectors per thread in flight in the element loops (measured on GB300: +0.7-1.5% with
  // bf16 dlogits, within +-0.4% with f32 dlogits, where a forced 1 was 1% slower).
  constexpr int kUnroll = 2;
  extern __shared__ __align__(128) unsigned char smem[];
  const int buf_bytes = (int)align_up((size_t)a.slice * sizeof(InT), 128);
  InT* buf = reinterpret_cast<InT*>(smem);
  const uint4* buf4 = reinterpret_cast<const uint4*>(smem);
  uint4* buf4w = reinterpret_cast<uint4*>(smem);  // kAny: realigned vectors are written here
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + buf_bytes);  // chunk k landed
  uint64_t* empty = full + a.n_chunks;                              // chunk k released
  uint64_t* xbars = empty + a.n_chunks;                             // 2 exchange barriers
  int* abort_flag = reinterpret_cast<int*>(xbars + 2);
  RowIn* rin = reinterpret_cast<RowIn*>(reinterpret_cast<unsigned char*>(abort_flag) + 16);
  float2* exch = reinterpret_cast<float2*>(rin + 2);                // [2][C * kWarps]

  // The fixed-order sum that follows (a programmatic dependent) may be scheduled now: it waits
  // for this grid to complete before it reads anything.
  allow_dependent_launch();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t rank = cluster_ctarank();
  const uint32_t C = cluster_nctarank();
  const int n_ent = (int)C * kWarps;  // exchange entries per row: one per warp of the cluster
  const int64_t ncl = cluster_count_x();
  const int s0 = (int)rank * a.slice;
  const int len = max(0, min(a.V - s0, a.slice));  // my slice's elements
  const int nvec = (kAny || a.bulk) ? len / kVec : 0;  // vectors (by bulk copy, or realigned)
  const int tail0 = nvec * kVec;                   // first element loaded one by one
  const uint32_t buf_s = smem_addr(buf);
  const uint32_t full_s = smem_addr(full), empty_s = smem_addr(empty);
  const uint32_t xbar_s = smem_addr(xbars), exch_s = smem_addr(exch);
  const float2 l2e2 = make_float2(kLog2e, kLog2e);
  // The layout (slice, barriers, row slots, exchange entries) within the launch's shared memory;
  // the same answer in every CTA of the cluster, which then only keeps the cluster barriers.
  if (!GRPO_DCHECK(reinterpret_cast<const unsigned char*>(exch + 2 * n_ent) - smem <=
                   (int64_t)dynamic_smem_bytes())) {
    __syncthreads();
    cluster_sync();
    __syncthreads();
    cluster_sync();
    return;
  }

  if (tid == 0) {
    for (int k = 0; k < a.n_chunks; ++k) {
      mbar_init(full_s + 8 * k, 1);
      mbar_init(empty_s + 8 * k, kWarps);
    }
    mbar_init(xbar_s, 1);
    mbar_init(xbar_s + 8, 1);
    *abort_flag = 0;
    for (int k = 0; k < 2; ++k) {  // a slot read after an abort names row 0 and no token
      rin[k].src = 0;
      rin[k].y = -1;
      rin[k].zy = rin[k].A = rin[k].old_lp = rin[k].ref_lp = rin[k].w = 0.f;
    }
    mbar_fence_init();
  }
  __syncthreads();
  cluster_sync();  // peers' exchange barriers exist before anyone sends to them

  int64_t n_rows = a.n_rows;
  double inv_denom = a.inv_denom;
  float inv_denom_f = a.inv_denom_f, inv_nseq_f = a.inv_nseq_f;
  if (a.counts) {
    const int64_t k_kept = a.counts[0], t_kept = a.counts[1];
    n_rows = t_kept < n_rows ? t_kept : n_rows;
    if (a.denom_from_counts) {
      inv_denom = t_kept > 0 ? 1.0 / (double)t_kept : 0.0;
      inv_denom_f = (float)inv_denom;
      inv_nseq_f = k_kept > 0 ? (float)(1.0 / (double)k_kept) : 0.f;
    }
  }

  // Bounded wait (about kWaitLimitNs).  A copy that never lands sets GRPO_DEVFLAG_TIMEOUT and
  // the abort flag, after which the CTA stops waiting for and issuing copies (its results are
  // then invalid) but still completes every exchange and chunk release, so that no peer writes
  // into a CTA that left and every wait of the producer ends.
  auto wait_bar = [&](uint32_t bar, uint32_t parity, bool copy) -> bool {  // true: phase done
    if (copy && *(volatile int*)abort_flag) return false;
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1; !mbar_try_wait(bar, parity); ++it) {
      if ((it & 63u) != 0) continue;
      if (copy && *(volatile int*)abort_flag) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *(volatile int*)abort_flag = 1;
        if (a.status) atomicOr(a.status, GRPO_DEVFLAG_TIMEOUT);
        return false;
      }
    }
    return true;
  };

  if (warp == kWarps) {
    // ---- producer warp, one lane: each row's inputs and its slice's copies ----
    if (lane == 0) {
      // Copies issued whose completion no consumer may have waited for (bit k: chunk k, with the
      // phase parity in pend_par); drained before the CTA exits.
      uint32_t pend = 0, pend_par = 0;
      auto fetch = [&](int64_t r) {
        RowIn ri;
        ri.src = a.row_index ? a.row_index[r] : r;
        if (!GRPO_DCHECK(ri.src >= 0)) ri.src = 0;
        ri.y = a.y[ri.src];
        ri.zy = (ri.y >= 0 && ri.y < a.V)
                    ? Fmt<InT>::load(reinterpret_cast<const InT*>(a.logits + ri.src * a.row_stride_bytes) + ri.y)
                    : 0.f;
        int32_t ro = a.row_rollout[r];
        if (!GRPO_DCHECK(ro >= 0)) ro = 0;
        ri.A = a.adv[ro];
        ri.old_lp = a.old_logp[ri.src];
        ri.ref_lp = a.ref_logp[ri.src];
        ri.w = a.agg_mode == 0 ? inv_denom_f
                               : inv_nseq_f / (float)(a.seq_off[ro + 1] - a.seq_off[ro]);
        return ri;
      };
      auto issue = [&](int64_t src, int k, uint32_t parity) {
        const char* g = a.logits + src * a.row_stride_bytes + (int64_t)s0 * sizeof(InT);
        const int v0 = k * a.chunk_vecs;
        const int v1 = min(nvec, v0 + a.chunk_vecs);
        uint32_t bytes = v1 > v0 ? (uint32_t)(v1 - v0) * 16u : 0u;
        if (kAny && (reinterpret_cast<uintptr_t>(g) & 15u)) bytes = 0;  // the consumers realign
        // a bulk copy needs 16-byte aligned addresses and a size in 16-byte units
        if (bytes && !GRPO_DCHECK(((reinterpret_cast<uintptr_t>(g) + (uintptr_t)v0 * 16) & 15u) == 0 &&
                                  v1 * 16 <= buf_bytes))
          bytes = 0;
        mbar_expect_tx(full_s + 8 * k, bytes);  // also publishes rin[] writes made before it
        if (bytes) bulk_copy_g2s(buf_s + v0 * 16, g + (int64_t)v0 * 16, bytes, full_s + 8 * k);
        pend |= 1u << k;
        pend_par = (pend_par & ~(1u << k)) | (parity << k);
      };
      int64_t row = cluster_id_x();
      RowIn nxt = {};
      if (row < n_rows) {
        rin[0] = fetch(row);
        for (int k = 0; k < a.n_chunks; ++k) {
          if (a.skip_copy && k == 0 && row == 0 && rank == 0) {  // test hook: arm, never copy
            mbar_expect_tx(full_s, 16u);
            pend |= 1u;
            continue;
          }
          issue(rin[0].src, k, 0u);
        }
        if (row + ncl < n_rows) nxt = fetch(row + ncl);  // loads in flight until it is needed
      }
      for (uint32_t iter = 0; row < n_rows; row += ncl, ++iter) {
        const uint32_t slot = iter & 1u;
        // one 8-byte entry from every warp of the cluster
        mbar_expect_tx(xbar_s + 8 * slot, 8u * (uint32_t)n_ent);
        const int64_t next = row + ncl;
        if (kAny && next < n_rows && nvec > 0 && !*(volatile int*)abort_flag) {
          // The consumers will realign the next row's slice with plain loads if it is not
          // 16-byte aligned: start its aligned interior on its way into L2 a row ahead.
          const uintptr_t g = reinterpret_cast<uintptr_t>(a.logits + nxt.src * a.row_stride_bytes) +
                              (uintptr_t)s0 * sizeof(InT);
          const uintptr_t lo = (g + 15u) & ~(uintptr_t)15u, hi = (g + (uintptr_t)nvec * 16u) & ~(uintptr_t)15u;
          if ((g & 15u) && hi > lo) bulk_prefetch_l2(reinterpret_cast<const void*>(lo), (uint32_t)(hi - lo));
        }
        for (int k = 0; k < a.n_chunks; ++k) {
          wait_bar(empty_s + 8 * k, iter & 1u, false);  // chunk k of this row is released
          if (next >= n_rows) continue;
          if (k == 0) rin[slot ^ 1u] = nxt;  // the consumers are done with the row before this one
          if (!*(volatile int*)abort_flag) issue(nxt.src, k, (iter + 1u) & 1u);
        }
        // The row after next: its dependent loads (source row, then token and log-probs) overlap
        // the consumers' pass A of the next row instead of delaying a refill.
        if (next + ncl < n_rows) nxt = fetch(next + ncl);
      }
      for (int k = 0; k < a.n_chunks; ++k)  // copies in flight land before the CTA exits
        if ((pend >> k) & 1u) wait_bar(full_s + 8 * k, (pend_par >> k) & 1u, false);
    }
    __syncwarp();
  } else {
    // ---- consumer warps ----
    int64_t row = cluster_id_x();
    for (uint32_t iter = 0; row < n_rows; row += ncl, ++iter) {
      const uint32_t slot = iter & 1u, phase = iter & 1u;
      RowIn ri = {};
      bool live = true;  // every chunk of this row arrived (no abort)
      int yl = -1;
      const char* grow = nullptr;
      int mis = 0;  // kAny: the slice's offset from a 16-byte boundary (0: it came by bulk copy)

      // ---- pass A: max and sum of exp over my elements, y left out ----
      float m = -INFINITY, s = 0.f;
      for (int k = 0; k < a.n_chunks; ++k) {
        if (!wait_bar(full_s + 8 * k, phase, true)) live = false;
        if (k == 0) {
          ri = rin[slot];
          const bool yv_ok = ri.y >= 0 && ri.y < a.V;
          yl = yv_ok ? ri.y - s0 : -1;  // y's position in my slice, if there
          grow = a.logits + ri.src * a.row_stride_bytes + (int64_t)s0 * sizeof(InT);
          if (kAny) mis = (int)(reinterpret_cast<uintptr_t>(grow) & 15u);
        }
        const int v0 = k * a.chunk_vecs;
        const int v1 = min(nvec, v0 + a.chunk_vecs);
        const bool last = (k == a.n_chunks - 1);
        typename Fmt<InT>::Max mx;
        if (kAny && mis) {
          // Vector j of the slice is bytes [mis, mis + 16) of aligned words j and j + 1 counted
          // from grow - mis; as row vector J = s0 / kVec + j those words lie inside the row when
          // 16 J >= mis (J >= 1) and 16 (J + 2) <= V * sizeof(InT) + mis: j in [jlo, jhi).  The
          // thread that owns vector j (j = v0 + tid mod kThreads) assembles it as in the aligned
          // instance; the maximum is exact, so the few vectors outside [jlo, jhi) (element by
          // element) go first and the rest in a loop without branches.
          const uint4* w16 = reinterpret_cast<const uint4*>(grow - mis);
          const int J0 = s0 / kVec;
          const int jlo = max(v0, 1 - J0);
          const int64_t jrow = (((int64_t)a.V * (int64_t)sizeof(InT) + mis) >> 4) - 1 - J0;
          const int jhi = jrow < (int64_t)v1 ? (int)jrow : v1;
          auto owned_from = [&](int start) {  // this thread's first vector at or after start
            const int j = v0 + tid;
            return j >= start ? j : j + (start - j + kThreads - 1) / kThreads * kThreads;
          };
          auto by_elements = [&](int j) {
            if (live) {  // after an abort nothing is read from global memory
              const InT* src = reinterpret_cast<const InT*>(grow) + j * kVec;
#pragma unroll
              for (int i = 0; i < kVec; ++i) buf[j * kVec + i] = src[i];
            }
            mx.add(buf4[j]);
          };
          for (int j = v0 + tid; j < min(v1, jlo); j += kThreads) by_elements(j);
          for (int j = owned_from(max(jlo, jhi)); j < v1; j += kThreads) by_elements(j);
          if (live) {
            // one loop per word offset (mis / 4, a compile-time constant of the loop)
            const uint32_t bsh = (uint32_t)(mis & 3) * 8u;
            auto realign = [&](auto qc) {
              constexpr int Q = decltype(qc)::value;
#pragma unroll 4
              for (int j = owned_from(jlo); j < jhi; j += kThreads) {
                const uint4 q = extract16_q<Q>(__ldcs(w16 + j), __ldcs(w16 + j + 1), bsh);
                buf4w[j] = q;
                mx.add(q);
              }
            };
            switch (mis >> 2) {
              case 0: realign(std::integral_constant<int, 0>{}); break;
              case 1: realign(std::integral_constant<int, 1>{}); break;
              case 2: realign(std::integral_constant<int, 2>{}); break;
              default: realign(std::integral_constant<int, 3>{}); break;
            }
          } else {
            for (int j = owned_from(jlo); j < jhi; j += kThreads) mx.add(buf4[j]);
          }
        } else {
#pragma unroll 4
          for (int j = v0 + tid; j < v1; j += kThreads) mx.add(buf4[j]);
        }
        float cm = mx.get();
        if (last) {
          for (int e = tail0 + tid; e < len; e += kThreads) {
            // after an abort the row inputs may be stale: nothing is read from global memory
            if (live) buf[e] = *reinterpret_cast<const InT*>(grow + (int64_t)e * sizeof(InT));
            cm = fmaxf(cm, Fmt<InT>::load(&buf[e]));  // read back below and in pass B
          }
        }
        if (cm > m) {
          s = (m == -INFINITY) ? 0.f : s * ex2((m - cm) * kLog2e);
          m = cm;
        }
        if (m != -INFINITY) {
          const float sh = -m * kLog2e;
          const float2 sh2 = make_float2(sh, sh);
          float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll kUnroll
          for (int j = v0 + tid; j < v1; j += kThreads) {
            float2 p[kPairs];
            Fmt<InT>::pairs(buf4[j], p);
            const int yi = yl - j * kVec;
            if ((unsigned)yi < (unsigned)kVec) {  // the vector holding y: leave y out
#pragma unroll
              for (int i = 0; i < kPairs; ++i) {
                const float2 e = ex2x2(__ffma2_rn(p[i], l2e2, sh2));
                if (2 * i != yi) acc0.x += e.x;
                if (2 * i + 1 != yi) acc0.y += e.y;
              }
            } else {
#pragma unroll
              for (int i = 0; i < kPairs; i += 2) {
                acc0 = __fadd2_rn(acc0, ex2x2(__ffma2_rn(p[i], l2e2, sh2)));
                acc1 = __fadd2_rn(acc1, ex2x2(__ffma2_rn(p[i + 1], l2e2, sh2)));
              }
            }
          }
          s += (acc0.x + acc0.y) + (acc1.x + acc1.y);
          if (last)
            for (int e = tail0 + tid; e < len; e += kThreads)
              if (e != yl) s += ex2(fmaf(Fmt<InT>::load(&buf[e]), kLog2e, sh));
        }
      }
      // warp reduction of (m, s); this warp's entry goes to every CTA of the cluster (self too)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float mo = __shfl_xor_sync(0xffffffffu, m, o);
        const float so = __shfl_xor_sync(0xffffffffu, s, o);
        lse_combine(m, s, mo, so);
      }
      if (lane < (int)C) {
        const uint32_t dst = exch_s + (uint32_t)(slot * n_ent + rank * kWarps + warp) * 8u;
        st_async_f2(mapa_shared(dst, lane), make_float2(m, s), mapa_shared(xbar_s + 8 * slot, lane));
      }

      // ---- exchange: this warp combines the cluster's entries and forms the row scalars ----
      wait_bar(xbar_s + 8 * slot, (iter >> 1) & 1u, false);
      const float2* ex = exch + slot * n_ent;
      float M = -INFINITY;
      for (int e = lane; e < n_ent; e += 32) M = fmaxf(M, ex[e].x);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      float S_excl = 0.f;
      for (int e = lane; e < n_ent; e += 32) {
        const float2 v = ex[e];
        if (v.x != -INFINITY) S_excl += v.y * expf(v.x - M);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) S_excl += __shfl_xor_sync(0xffffffffu, S_excl, o);
      const bool yvalid = ri.y >= 0 && ri.y < a.V;
      const bool writer = rank == 0 && warp == 0 && lane == 0;
      float neg_scale = 0.f, dy = 0.f, shB = 0.f;
      if (!yvalid) {
        if (writer) {
          if (a.logp_out) a.logp_out[row] = __int_as_float(0x7fc00000);
          a.row_loss[row] = 0.0;
          if (a.status) atomicOr(a.status, GRPO_DEVFLAG_BAD_TOKEN);
        }
      } else {
        const float zy = ri.zy;
        const float ey = expf(zy - M);
        const float S = S_excl + ey;
        const float logp = (zy - M) - logf(S);
        // Eq. 1: ratio, clipped surrogate, KL term; Eqs. 2-3: gradient coefficient.
        const float A = ri.A;
        const float rho = expf(logp - ri.old_lp);
        const float clipped = rho < a.lo_up ? a.lo_rn : (rho > a.hi_dn ? a.hi_rn : rho);
        const float surr = fminf(rho * A, clipped * A);
        const float x = ri.ref_lp - logp;
        const float em1 = expm1f(x);
        const float kl = em1 - x;
        const float ell = -(surr - a.beta * kl);
        const bool c = (A >= 0.f) ? (rho <= a.hi_dn) : (rho >= a.lo_up);
        const float g = -((c ? rho * A : 0.f) + a.beta * em1);
        const float coef = ri.w * g;
        neg_scale = -coef / S;
        dy = coef * (S_excl / S);
        shB = -M * kLog2e;
        if (fabsf(neg_scale) >= 0x1p-100f) {
          shB += kShiftB;
          neg_scale *= 0x1p-16f;  // 2^-kShiftB
        }
        if (writer) {
          if (a.logp_out) a.logp_out[row] = logp;
          a.row_loss[row] = (a.agg_mode == 0 ? inv_denom : (double)ri.w) * (double)ell;
          if (a.status && !isfinite(logp)) atomicOr(a.status, GRPO_DEVFLAG_NONFINITE);
        }
      }

      // ---- pass B: dlogits from the shared-memory slice; each chunk released when done ----
      const float2 shb2 = make_float2(shB, shB), ns2 = make_float2(neg_scale, neg_scale);
      OutT* orow = reinterpret_cast<OutT*>(a.dlogits) + row * (int64_t)a.V + s0;
      const int omis = kAny ? (int)(reinterpret_cast<uintptr_t>(orow) & 15u) : 0;
      if (kAny) {
        // This thread's plain stores into the slice (realigned vectors, elements) come before
        // any later bulk copy into it (the async proxy), and every consumer's pass-A stores are
        // visible to every consumer.
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("bar.sync 1, %0;" ::"r"(kThreads) : "memory");
      }
      if (kAny && omis) {
        // Aligned 16-byte output words: word w holds slice elements [h + w E, h + (w + 1) E);
        // the first h and the last (len - h) % E elements are stored one by one.  Each word and
        // element is written in the iteration of the chunk that holds its first input byte, and
        // chunk k is released after its iteration: later iterations read only later chunks.
        using OW = OutWord<InT, OutT>;
        constexpr int E = OW::kElems;
        const int h = min(len, ((16 - omis) & 15) / (int)sizeof(OutT));
        const int nfull = (len - h) / E;
        const int rest0 = h + nfull * E;
        const int chunk_elems = a.chunk_vecs * kVec;
        auto chunk_of = [&](int e) { return min(e / chunk_elems, a.n_chunks - 1); };
        int w_begin = 0;
        for (int k = 0; k < a.n_chunks; ++k) {
          // the words whose first element lies in chunks <= k
          int w_end = nfull;
          if (k < a.n_chunks - 1) {
            const int e_next = (k + 1) * chunk_elems;  // first element of chunk k + 1
            w_end = e_next <= h ? 0 : min(nfull, (e_next - h + E - 1) / E);
          }
          for (int w = w_begin + tid; w < w_end; w += kThreads) {
            const int i0 = h + w * E;
            float2 d[OW::kPairs];
            if (yvalid &&
                GRPO_DCHECK((i0 * (int)sizeof(InT) + OW::kInBytes + 15) / 16 * 16 <= buf_bytes)) {
              float2 p[OW::kPairs];
              pairs_at<InT, OutT>(buf4, i0, p);
#pragma unroll
              for (int i = 0; i < OW::kPairs; ++i)
                d[i] = __fmul2_rn(ex2x2(__ffma2_rn(p[i], l2e2, shb2)), ns2);
              const int yi = yl - i0;
              if ((unsigned)yi < (unsigned)E) {
#pragma unroll
                for (int i = 0; i < OW::kPairs; ++i) {
                  if (2 * i == yi) d[i].x = dy;
                  if (2 * i + 1 == yi) d[i].y = dy;
                }
              }
            } else {
#pragma unroll
              for (int i = 0; i < OW::kPairs; ++i) d[i] = make_float2(0.f, 0.f);
            }
            store_pairs<OutT, OW::kPairs>(orow + i0, d);
          }
          w_begin = max(w_begin, w_end);
          for (int t = tid; t < h + (len - rest0); t += kThreads) {
            const int e = t < h ? t : rest0 + (t - h);  // the head, then the tail
            if (chunk_of(e) != k) continue;
            float d = 0.f;
            if (yvalid) {
              d = neg_scale * ex2(fmaf(Fmt<InT>::load(&buf[e]), kLog2e, shB));
              if (e == yl) d = dy;
            }
            Fmt<OutT>::store(orow + e, d);
          }
          __syncwarp();  // every lane of this warp is done reading chunk k
          if (lane == 0) mbar_arrive(empty_s + 8 * k);
        }
        continue;
      }
      for (int k = 0; k < a.n_chunks; ++k) {
        const int v0 = k * a.chunk_vecs;
        const int v1 = min(nvec, v0 + a.chunk_vecs);
        const bool last = (k == a.n_chunks - 1);
        if (yvalid) {
#pragma unroll kUnroll
          for (int j = v0 + tid; j < v1; j += kThreads) {
            float2 p[kPairs], d[kPairs];
            Fmt<InT>::pairs(buf4[j], p);
#pragma unroll
            for (int i = 0; i < kPairs; ++i)
              d[i] = __fmul2_rn(ex2x2(__ffma2_rn(p[i], l2e2, shb2)), ns2);
            const int yi = yl - j * kVec;
            if ((unsigned)yi < (unsigned)kVec) {
#pragma unroll
              for (int i = 0; i < kPairs; ++i) {
                if (2 * i == yi) d[i].x = dy;
                if (2 * i + 1 == yi) d[i].y = dy;
              }
            }
            if (kAny || a.out_vec)  // (kAny reaches this loop only for a 16-byte aligned row)
              store_pairs<OutT, kPairs>(orow + j * kVec, d);
            else
              store_pairs_scalar<OutT, kPairs>(orow + j * kVec, d);
          }
          if (last) {
            for (int e = tail0 + tid; e < len; e += kThreads) {
              float d = neg_scale * ex2(fmaf(Fmt<InT>::load(&buf[e]), kLog2e, shB));
              if (e == yl) d = dy;
              Fmt<OutT>::store(orow + e, d);
            }
          }
        } else {
          float2 d[kPairs];
#pragma unroll
          for (int i = 0; i < kPairs; ++i) d[i] = make_float2(0.f, 0.f);
          for (int j = v0 + tid; j < v1; j += kThreads)
            store_pairs_scalar<OutT, kPairs>(orow + j * kVec, d);
          if (last)
            for (int e = tail0 + tid; e < len; e += kThreads) Fmt<OutT>::store(orow + e, 0.f);
        }
        __syncwarp();  // every lane of this warp is done reading chunk k
        if (lane == 0) mbar_arrive(empty_s + 8 * k);
      }
    }
  }
  __syncthreads();
  cluster_sync();  // partners are done with this CTA's shared memory
}


// ---- forward only: log-probabilities (and softmax statistics) as a plain stream ---------------
//
// Without a gradient pass there is nothing to keep in shared memory, so a row needs no cluster:
// one CTA streams the whole row with kU independent 16-byte loads per thread in flight, keeps an
// online (max, sum of exp) leaving y out, and reduces it across the CTA.  The grid is persistent
// and never larger than what can be resident (with more CTAs than fit, the rest would wait for
// a whole second pass); 1536 resident threads per SM.  Measured on GB300: ~7.1 TB/s on the qwen
// rows, 98% of a read-only stream, against 6.6 TB/s for the cluster kernel without pass B.
constexpr int kFwdThreads = 128;
constexpr int kFwdUnroll = 4;
constexpr int kFwdResident = 1536;

template <typename InT, bool kAny>
__global__ void __launch_bounds__(kFwdThreads, kFwdResident / kFwdThreads)
    logp_stream_kernel(const LossArgs a) {
  constexpr int kVec = Fmt<InT>::kVec;
  constexpr int kPairs = Fmt<InT>::kPairs;
  constexpr int kWarps = kFwdThreads / 32;
  constexpr int kSeg = kFwdThreads * kFwdUnroll;
  __shared__ float red[2 * kWarps];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nvec = (kAny || a.bulk) ? a.V / kVec : 0;
  const int tail0 = nvec * kVec;
  const float2 l2e2 = make_float2(kLog2e, kLog2e);
  int64_t n_rows = a.n_rows;
  if (a.counts && a.counts[1] < n_rows) n_rows = a.counts[1];  // device count of kept rows
  for (int64_t row = blockIdx.x; row < n_rows; row += gridDim.x) {
    int64_t src = a.row_index ? a.row_index[row] : row;
    if (!GRPO_DCHECK(src >= 0)) src = 0;
    const int32_t yv = a.y[src];
    const bool yvalid = yv >= 0 && yv < a.V;
    const int yl = yvalid ? yv : -1;
    const InT* grow = reinterpret_cast<const InT*>(a.logits + src * a.row_stride_bytes);
    const uint4* g4 = reinterpret_cast<const uint4*>(grow);
    // kAny (rows that need not start on a 16-byte boundary): each vector from the aligned words
    // that hold it (vec_at_global)
    const int mis = kAny ? (int)(reinterpret_cast<uintptr_t>(grow) & 15u) : 0;
    float m = -INFINITY, s = 0.f;  // running max and sum of exp(z - m), y left out
    for (int jb = 0; jb < nvec; jb += kSeg) {
      uint4 q[kFwdUnroll];
#pragma unroll
      for (int u = 0; u < kFwdUnroll; ++u) {
        const int j = jb + u * kFwdThreads + tid;
        if (j < nvec) q[u] = kAny ? vec_at_global(grow, mis, a.V, j) : __ldcs(g4 + j);
      }
      typename Fmt<InT>::Max mx;
#pragma unroll
      for (int u = 0; u < kFwdUnroll; ++u)
        if (jb + u * kFwdThreads + tid < nvec) mx.add(q[u]);
      const float cm = mx.get();
      if (cm > m) {
        s = (m == -INFINITY) ? 0.f : s * ex2((m - cm) * kLog2e);
        m = cm;
      }
      if (m == -INFINITY) continue;
      const float sh = -m * kLog2e;
      const float2 sh2 = make_float2(sh, sh);
      float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
      for (int u = 0; u < kFwdUnroll; ++u) {
        const int j = jb + u * kFwdThreads + tid;
        if (j >= nvec) continue;
        float2 p[kPairs];
        Fmt<InT>::pairs(q[u], p);
        const int yi = yl - j * kVec;
        if ((unsigned)yi < (unsigned)kVec) {  // the vector holding y: leave y out
#pragma unroll
          for (int i = 0; i < kPairs; ++i) {
            const float2 e = ex2x2(__ffma2_rn(p[i], l2e2, sh2));
            if (2 * i != yi) acc0.x += e.x;
            if (2 * i + 1 != yi) acc0.y += e.y;
          }
        } else {
#pragma unroll
          for (int i = 0; i < kPairs; i += 2) {
            acc0 = __fadd2_rn(acc0, ex2x2(__ffma2_rn(p[i], l2e2, sh2)));
            acc1 = __fadd2_rn(acc1, ex2x2(__ffma2_rn(p[i + 1], l2e2, sh2)));
          }
        }
      }
      s += (acc0.x + acc0.y) + (acc1.x + acc1.y);
    }
    for (int e = tail0 + tid; e < a.V; e += kFwdThreads) {  // ragged tail
      const float v = Fmt<InT>::load(grow + e);
      if (v > m) {
        s = (m == -INFINITY) ? 0.f : s * ex2((m - v) * kLog2e);
        m = v;
      }
      if (e != yl) s += ex2((v - m) * kLog2e);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float mo = __shfl_xor_sync(0xffffffffu, m, o);
      const float so = __shfl_xor_sync(0xffffffffu, s, o);
      lse_combine(m, s, mo, so);
    }
    if (lane == 0) {
      red[2 * warp] = m;
      red[2 * warp + 1] = s;
    }
    __syncthreads();
    if (warp == 0) {
      m = lane < kWarps ? red[2 * lane] : -INFINITY;
      s = lane < kWarps ? red[2 * lane + 1] : 0.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float mo = __shfl_xor_sync(0xffffffffu, m, o);
        const float so = __shfl_xor_sync(0xffffffffu, s, o);
        lse_combine(m, s, mo, so);
      }
      if (lane == 0) {
        if (!yvalid) {
          a.logp_out[row] = __int_as_float(0x7fc00000);
          if (a.stats_out) a.stats_out[row] = make_float4(NAN, NAN, NAN, 0.f);
          if (a.status) atomicOr(a.status, GRPO_DEVFLAG_BAD_TOKEN);
        } else {
          const float zy = Fmt<InT>::load(grow + yv);
          const float S = s + expf(zy - m);
          const float logp = (zy - m) - logf(S);
          a.logp_out[row] = logp;
          if (a.stats_out) a.stats_out[row] = make_float4(m, S, s, 0.f);
          if (a.status && !isfinite(logp)) atomicOr(a.status, GRPO_DEVFLAG_NONFINITE);
        }
      }
    }
    __syncthreads();  // red[] is reused by the next row
  }
}

// ---- host side --------------------------------------------------------------------------------

struct Tune {
  int cluster = 0, threads = 0, chunks = 0;
};
Tune g_tune;
std::mutex g_mu;
std::atomic<int> g_skip_copy{0};
std::map<std::tuple<const void*, int, int, int>, int> g_max_clusters;  // (kernel, dev, C, smem)
std::map<std::pair<const void*, int>, size_t> g_smem_attr;            // (kernel, dev) -> bytes set
std::map<std::pair<const void*, int>, int> g_resident_ctas;            // (kernel, dev) -> CTAs

using KernelFn = void (*)(LossArgs);

template <typename InT, typename OutT, bool kCap, bool kAny>
KernelFn pick_threads(int threads) {
  switch (threads) {
    case 128: return grpo_loss_kernel<InT, OutT, 128, kCap, kAny>;
    case 512: return grpo_loss_kernel<InT, OutT, 512, kCap, kAny>;
    default: return grpo_loss_kernel<InT, OutT, 256, kCap, kAny>;
  }
}

// any: rows of logits or dlogits that need not start on a 16-byte boundary (the kAny instance,
// compiled without the register cap).
template <typename InT, typename OutT>
KernelFn pick_kernel(int threads, bool cap, bool any) {
  if (any) return pick_threads<InT, OutT, false, true>(threads);
  return cap ? pick_threads<InT, OutT, true, false>(threads)
             : pick_threads<InT, OutT, false, false>(threads);
}

KernelFn kernel_for(int in_dtype, int out_dtype, int threads, bool cap, bool any) {
  if (in_dtype == GRPO_DTYPE_BF16)
    return out_dtype == GRPO_DTYPE_BF16 ? pick_kernel<__nv_bfloat16, __nv_bfloat16>(threads, cap, any)
                                        : pick_kernel<__nv_bfloat16, float>(threads, cap, any);
  return out_dtype == GRPO_DTYPE_BF16 ? pick_kernel<float, __nv_bfloat16>(threads, cap, any)
                                      : pick_kernel<float, float>(threads, cap, any);
}

// Whether shared memory would let more CTAs of this shape reside on an SM than the uncapped
// instance is compiled for (then the register-capped instance keeps that occupancy).
bool want_cap(size_t smem, int threads) {
  const size_t per_sm = 228 * 1024, reserved = 1024;
  return per_sm / (smem + reserved) > (size_t)uncapped_ctas(threads);
}

// Launch shape of the row kernel for a vocabulary of V entries of in_bytes each.
struct Shape {
  int C = 1, threads = 256, slice = 0, chunk_vecs = 0, chunks = 1;
  size_t smem = 0;
};

// out_bytes: bytes per dlogits element (2 or 4).
//
// Default shape, from sweeps on GB300 of every cluster size 1-16, 128/256/512 consumer threads
// and 1-3 copies per slice at V = 32000 ... 256000 (11 vocabularies), bf16 logits, bf16 and f32
// dlogits, about 12 GB per call:
//  - dlogits no wider than the logits: the cluster size C <= 10 that keeps the most slice bytes
//    resident per SM (CTAs per SM by shared memory, at most the CTAs the instance is compiled
//    for, times the slice's bytes), slices of at most 100 KiB; among sizes within 2% of the
//    most, the smallest.  256 consumer threads for slices of 56 KiB or more, else 128.  The
//    shape it picks was within 1% of the best measured one at every vocabulary but V = 32000
//    (2%, run-to-run noise on the same shape); the previous rule (80 KiB slices) left 9-16% at
//    V = 128256 and 201088;
//  - f32 dlogits from bf16 logits (the write phase twice the read): slices of about 24 KiB
//    (C = ceil(row / 24 KiB), at most 8), more CTAs per row while a slice exceeds 52 KiB (up to
//    10), 128 threads: within 1.6% of the best at every vocabulary, up to 18% above the
//    previous rule (40 KiB slices);
//  - two copies per slice, but one for slices of at most 32 KiB with narrow dlogits.
// Rows too long for those limits take up to 16 CTAs and slices up to the shared-memory limit.
grpo_status pick_shape(int V, int in_bytes, int out_bytes, const char* who, Shape* out) {
  Tune tune;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    tune = g_tune;
  }
  const int vec = 16 / in_bytes;
  const bool wide_out = out_bytes > in_bytes;
  auto slice_of = [&](int C) { return (int)align_up((size_t)((V + C - 1) / C), vec); };
  auto empty_slice = [&](int C) { return C > 1 && (int64_t)(C - 1) * slice_of(C) >= V; };
  auto threads_for = [&](int slice) {
    return (!wide_out && (size_t)slice * in_bytes >= 56 * 1024) ? 256 : 128;
  };
  int C = tune.cluster;
  if (C == 0 && wide_out) {
    const int64_t row_bytes = (int64_t)V * in_bytes;
    C = (int)std::min<int64_t>(8, std::max<int64_t>(1, (row_bytes + 24 * 1024 - 1) / (24 * 1024)));
    while (C < kMaxCluster) {
      const size_t sb = (size_t)slice_of(C) * in_bytes;
      if (sb > 100 * 1024 || (C < 10 && sb > 52 * 1024))
        ++C;
      else
        break;
    }
  } else if (C == 0) {
    const size_t per_sm = 228 * 1024, reserved = 1024;
    for (int pass = 0; pass < 2 && C == 0; ++pass) {
      const int cmax = pass == 0 ? 10 : kMaxCluster;
      const size_t smax = pass == 0 ? 100 * 1024 : 227 * 1024;
      size_t score[kMaxCluster + 1] = {};
      size_t top = 0;
      for (int c = 1; c <= cmax; ++c) {
        const int sl = slice_of(c);
        const size_t sb = (size_t)sl * in_bytes;
        if (empty_slice(c) || sb > smax) continue;
        const int th = threads_for(sl);
        const size_t smem = align_up(sb, 128) + loss_smem_fixed(2) + 2 * (size_t)c * (th / 32) * sizeof(float2);
        const size_t ctas = std::min<size_t>(per_sm / (smem + reserved), (size_t)uncapped_ctas(th));
        score[c] = ctas * sb;
        top = std::max(top, score[c]);
      }
      for (int c = 1; c <= cmax && top > 0; ++c)
        if (score[c] > 0 && (double)score[c] >= 0.98 * (double)top) {
          C = c;
          break;
        }
    }
    if (C == 0) C = kMaxCluster;  // the shared-memory check below reports what does not fit
  }
  int slice = slice_of(C);
  while (C > 1 && empty_slice(C)) {  // no empty slices
    --C;
    slice = slice_of(C);
  }
  const int threads = tune.threads ? tune.threads : threads_for(slice);
  const size_t slice_bytes = (size_t)slice * in_bytes;
  int chunks = tune.chunks ? tune.chunks : ((!wide_out && slice_bytes <= 32 * 1024) ? 1 : 2);
  const int slice_vecs = slice / vec;
  int chunk_vecs = (slice_vecs + chunks - 1) / chunks;
  if (chunk_vecs < 1) chunk_vecs = 1;
  // whole vectors per thread in every chunk but the last one
  const int even = (chunk_vecs + threads - 1) / threads * threads;
  if (even <= slice_vecs) chunk_vecs = even;
  chunks = (slice_vecs + chunk_vecs - 1) / chunk_vecs;
  if (chunks < 1) chunks = 1;
  if (chunks > kMaxChunks) {
    chunk_vecs = (slice_vecs + kMaxChunks - 1) / kMaxChunks;
    chunks = (slice_vecs + chunk_vecs - 1) / chunk_vecs;
  }
  const size_t smem = align_up(slice_bytes, 128) + loss_smem_fixed(chunks) +
                      2 * (size_t)C * (threads / 32) * sizeof(float2);
  if (smem > 227 * 1024)
    return fail(GRPO_ERR_UNSUPPORTED, "%s: V = %d needs %zu bytes of shared memory per CTA at %d CTAs", who,
                V, smem, C);
  out->C = C;
  out->threads = threads;
  out->slice = slice;
  out->chunk_vecs = chunk_vecs;
  out->chunks = chunks;
  out->smem = smem;
  return GRPO_OK;
}

// Persistent cluster launch: as many clusters as can be resident, at most one per row.
grpo_status launch_rows(KernelFn fn, const Shape& sh, LossArgs a, cudaStream_t s, const char* who) {
  a.slice = sh.slice;
  a.chunk_vecs = sh.chunk_vecs;
  a.n_chunks = sh.chunks;
  cudaError_t e = cudaSuccess;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = sh.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(sh.threads + 32, 1, 1);  // consumers and the producer warp
  cfg.dynamicSmemBytes = sh.smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int dev = 0;
  cudaGetDevice(&dev);
  int max_cl = 0;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    const auto key = std::make_tuple((const void*)fn, dev, sh.C, (int)sh.smem);
    auto it = g_max_clusters.find(key);
    if (it != g_max_clusters.end()) {
      max_cl = it->second;
    } else {  // first launch of this kernel and shape on this device: set it up once
      size_t& have = g_smem_attr[std::make_pair((const void*)fn, dev)];
      if (sh.smem > have) {  // the attribute is a maximum: only ever raise it
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
        if (e == cudaSuccess) have = sh.smem;
      }
      if (e == cudaSuccess && sh.C > 8)
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "%s: cudaFuncSetAttribute: %s", who, cudaGetErrorString(e));
      cfg.gridDim = dim3(sh.C, 1, 1);
      e = cudaOccupancyMaxActiveClusters(&max_cl, fn, &cfg);
      if (e != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "%s: cudaOccupancyMaxActiveClusters: %s", who, cudaGetErrorString(e));
      if (max_cl < 1)
        return fail(GRPO_ERR_UNSUPPORTED, "%s: a cluster of %d CTAs with %zu bytes each cannot be resident",
                    who, sh.C, sh.smem);
      g_max_clusters[key] = max_cl;
    }
  }
  const int64_t n_clusters = std::min<int64_t>(a.n_rows, max_cl);
  cfg.gridDim = dim3((unsigned)(n_clusters * sh.C), 1, 1);
  e = cudaLaunchKernelEx(&cfg, fn, a);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: launch: %s", who, cudaGetErrorString(e));
  return GRPO_OK;
}

}  // namespace
}  // namespace fastrl

using namespace fastrl;

extern "C" grpo_status grpo_test_skip_copy(int32_t enable) {
  clear_error();
  g_skip_copy.store(enable ? 1 : 0);
  return GRPO_OK;
}

extern "C" grpo_status grpo_loss_tune(int32_t cluster_ctas, int32_t threads, int32_t chunks) {
  clear_error();
  if (cluster_ctas < 0 || cluster_ctas > kMaxCluster)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_loss_tune: cluster_ctas = %d", cluster_ctas);
  if (threads != 0 && threads != 128 && threads != 256 && threads != 512)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_loss_tune: threads = %d", threads);
  if (chunks < 0 || chunks > kMaxChunks)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_loss_tune: chunks = %d", chunks);
  std::lock_guard<std::mutex> lk(g_mu);
  g_tune.cluster = cluster_ctas;
  g_tune.threads = threads;
  g_tune.chunks = chunks;
  return GRPO_OK;
}


namespace fastrl {
namespace {

// The fused loss; counts (device {K, T_kept}, nullable) bounds the rows on the device and, with
// a non-positive denom_tokens / n_seq, supplies the token-mean denominator / sequence count.
grpo_status loss_impl(const char* who, const void* logits, int32_t logits_dtype, int64_t row_stride,
                      const int64_t* row_index, int64_t n_rows, const int64_t* counts, int32_t V,
                      const int32_t* y, const float* old_logp, const float* ref_logp,
                      const float* adv, const int32_t* row_rollout, float eps_low, float eps_high,
                      float beta, int32_t agg_mode, int64_t denom_tokens, const int64_t* seq_off,
                      int64_t n_seq, void* dlogits, int32_t dlogits_dtype, float* logp_out,
                      double* row_loss_out, double* loss_out, int32_t* status, void* ws,
                      size_t* ws_bytes, grpo_stream_t stream) {
  const bool from_counts = counts != nullptr && ((agg_mode == 0 && denom_tokens <= 0) ||
                                                 (agg_mode == 1 && n_seq <= 0));
  if (from_counts) {  // both denominators come from the device counts
    denom_tokens = 1;
    n_seq = 1;
  }
  if (logits_dtype != GRPO_DTYPE_BF16 && logits_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: logits_dtype = %d", who, logits_dtype);
  if (dlogits_dtype != GRPO_DTYPE_BF16 && dlogits_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: dlogits_dtype = %d", who, dlogits_dtype);
  if (n_rows < 0 || n_rows >= (int64_t(1) << 31))
    return fail(GRPO_ERR_INVALID_ARG, "%s: n_rows = %lld", who, (long long)n_rows);
  if (V < 1 || row_stride < V)
    return fail(GRPO_ERR_INVALID_ARG, "%s: V = %d, row_stride = %lld", who, V, (long long)row_stride);
  if (agg_mode != 0 && agg_mode != 1)
    return fail(GRPO_ERR_INVALID_ARG, "%s: agg_mode = %d", who, agg_mode);
  if (agg_mode == 0 && denom_tokens <= 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: denom_tokens = %lld", who, (long long)denom_tokens);
  if (agg_mode == 1 && (seq_off == nullptr || n_seq <= 0))
    return fail(GRPO_ERR_INVALID_ARG, "%s: agg_mode 1 needs seq_off and n_seq > 0", who);
  if (!(beta >= 0.f) || !(eps_low >= 0.f) || !(eps_high >= 0.f))
    return fail(GRPO_ERR_INVALID_ARG, "%s: beta, eps_low, eps_high must be >= 0", who);
  const size_t need = row_loss_out ? 0 : align_up((size_t)n_rows * 8, 256);
  bool query = false;
  grpo_status st = workspace_check(ws, ws_bytes, need, who, &query);
  if (st != GRPO_OK || query) return st;
  if (loss_out == nullptr) return fail(GRPO_ERR_INVALID_ARG, "%s: loss_out is NULL", who);
  double* row_loss = row_loss_out ? row_loss_out : static_cast<double*>(ws);
  cudaStream_t s = as_stream(stream);
  if (n_rows == 0) {
    return launch_sum_rows(row_loss, 0, nullptr, loss_out, s, who);
  }
  if (!logits || !y || !old_logp || !ref_logp || !adv || !row_rollout || !dlogits)
    return fail(GRPO_ERR_INVALID_ARG, "%s: NULL array", who);

  const int in_bytes = logits_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  const int out_bytes = dlogits_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  if (reinterpret_cast<uintptr_t>(logits) % in_bytes || reinterpret_cast<uintptr_t>(dlogits) % out_bytes)
    return fail(GRPO_ERR_INVALID_ARG, "%s: logits or dlogits not aligned to its element size", who);
  Shape sh;
  st = pick_shape(V, in_bytes, out_bytes, who, &sh);
  if (st != GRPO_OK) return st;

  LossArgs a = {};
  a.logits = static_cast<const char*>(logits);
  a.row_stride_bytes = row_stride * in_bytes;
  a.row_index = row_index;
  a.n_rows = n_rows;
  a.V = V;
  a.y = y;
  a.old_logp = old_logp;
  a.ref_logp = ref_logp;
  a.adv = adv;
  a.row_rollout = row_rollout;
  {
    const double lo = 1.0 - (double)eps_low, hi = 1.0 + (double)eps_high;
    const float lo_f = (float)lo, hi_f = (float)hi;  // nearest
    a.lo_rn = lo_f;
    a.hi_rn = hi_f;
    a.lo_up = (double)lo_f < lo ? std::nextafter(lo_f, INFINITY) : lo_f;
    a.hi_dn = (double)hi_f > hi ? std::nextafter(hi_f, -INFINITY) : hi_f;
  }
  a.beta = beta;
  a.agg_mode = agg_mode;
  a.inv_denom = agg_mode == 0 ? 1.0 / (double)denom_tokens : 0.0;
  a.inv_denom_f = (float)a.inv_denom;
  a.seq_off = seq_off;
  a.inv_nseq_f = agg_mode == 1 ? (float)(1.0 / (double)n_seq) : 0.f;
  a.dlogits = static_cast<char*>(dlogits);
  a.logp_out = logp_out;
  a.row_loss = row_loss;
  a.status = status;
  a.bulk = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && (a.row_stride_bytes % 16 == 0);
  a.out_vec = (reinterpret_cast<uintptr_t>(dlogits) % 16 == 0) && (((int64_t)V * out_bytes) % 16 == 0);
  a.counts = counts;
  a.denom_from_counts = from_counts ? 1 : 0;
  a.skip_copy = g_skip_copy.exchange(0);

  const bool any = !a.bulk || !a.out_vec;
  st = launch_rows(
      kernel_for(logits_dtype, dlogits_dtype, sh.threads, !any && want_cap(sh.smem, sh.threads), any),
      sh, a, s, who);
  if (st != GRPO_OK) return st;
  count_launches(1);
  return launch_sum_rows(row_loss, n_rows, counts ? counts + 1 : nullptr, loss_out, s, who);
}

}  // namespace
}  // namespace fastrl

extern "C" grpo_status grpo_loss_fwd_bwd(
    const void* logits, int32_t logits_dtype, int64_t row_stride, const int64_t* row_index,
    int64_t n_rows, int32_t V, const int32_t* y, const float* old_logp, const float* ref_logp,
    const float* adv, const int32_t* row_rollout, float eps_low, float eps_high, float beta,
    int32_t agg_mode, int64_t denom_tokens, const int64_t* seq_off, int64_t n_seq, void* dlogits,
    int32_t dlogits_dtype, float* logp_out, double* row_loss_out, double* loss_out, int32_t* status,
    void* ws, size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_loss_fwd_bwd");
  clear_error();
  return loss_impl("grpo_loss_fwd_bwd", logits, logits_dtype, row_stride, row_index, n_rows, nullptr,
                   V, y, old_logp, ref_logp, adv, row_rollout, eps_low, eps_high, beta, agg_mode,
                   denom_tokens, seq_off, n_seq, dlogits, dlogits_dtype, logp_out, row_loss_out,
                   loss_out, status, ws, ws_bytes, stream);
}

extern "C" grpo_status grpo_loss_fwd_bwd_dev(
    const void* logits, int32_t logits_dtype, int64_t row_stride, const int64_t* row_index,
    int64_t max_rows, const int64_t* counts, int32_t V, const int32_t* y, const float* old_logp,
    const float* ref_logp, const float* adv, const int32_t* row_rollout, float eps_low,
    float eps_high, float beta, int32_t agg_mode, int64_t denom_tokens, const int64_t* seq_off,
    int64_t n_seq, void* dlogits, int32_t dlogits_dtype, float* logp_out, double* row_loss_out,
    double* loss_out, int32_t* status, void* ws, size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_loss_fwd_bwd_dev");
  clear_error();
  if (counts == nullptr)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_loss_fwd_bwd_dev: counts is NULL");
  return loss_impl("grpo_loss_fwd_bwd_dev", logits, logits_dtype, row_stride, row_index, max_rows,
                   counts, V, y, old_logp, ref_logp, adv, row_rollout, eps_low, eps_high, beta,
                   agg_mode, denom_tokens, seq_off, n_seq, dlogits, dlogits_dtype, logp_out,
                   row_loss_out, loss_out, status, ws, ws_bytes, stream);
}


namespace fastrl {

grpo_status logp_rows(const char* who, const void* logits, int32_t logits_dtype, int64_t row_stride,
                      const int64_t* row_index, int64_t n_rows, const int64_t* counts, int32_t V,
                      const int32_t* y, float* logp_out, float4* stats_out, int32_t* status,
                      cudaStream_t s) {
  if (logits_dtype != GRPO_DTYPE_BF16 && logits_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: logits_dtype = %d", who, logits_dtype);
  if (n_rows < 0 || n_rows >= (int64_t(1) << 31))
    return fail(GRPO_ERR_INVALID_ARG, "%s: n_rows = %lld", who, (long long)n_rows);
  if (V < 1 || row_stride < V)
    return fail(GRPO_ERR_INVALID_ARG, "%s: V = %d, row_stride = %lld", who, V, (long long)row_stride);
  if (n_rows == 0) return GRPO_OK;
  if (!logits || !y || !logp_out) return fail(GRPO_ERR_INVALID_ARG, "%s: NULL array", who);
  const int in_bytes = logits_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  LossArgs a = {};
  a.logits = static_cast<const char*>(logits);
  a.row_stride_bytes = row_stride * in_bytes;
  a.row_index = row_index;
  a.n_rows = n_rows;
  a.V = V;
  a.y = y;
  a.logp_out = logp_out;
  a.stats_out = stats_out;
  a.status = status;
  a.counts = counts;
  a.bulk = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && (a.row_stride_bytes % 16 == 0);
  if (reinterpret_cast<uintptr_t>(logits) % in_bytes)
    return fail(GRPO_ERR_INVALID_ARG, "%s: logits not aligned to its element size", who);
  KernelFn fn = logits_dtype == GRPO_DTYPE_BF16
                    ? (a.bulk ? logp_stream_kernel<__nv_bfloat16, false> : logp_stream_kernel<__nv_bfloat16, true>)
                    : (a.bulk ? logp_stream_kernel<float, false> : logp_stream_kernel<float, true>);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: cudaGetDevice: %s", who, cudaGetErrorString(e));
  int resident = 0;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    const auto key = std::make_pair((const void*)fn, dev);
    auto it = g_resident_ctas.find(key);
    if (it != g_resident_ctas.end()) {
      resident = it->second;
    } else {  // resident CTAs on this device: every CTA of the persistent grid runs at once
      int per_sm = 0, sms = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kFwdThreads, 0);
      if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "%s: occupancy query: %s", who, cudaGetErrorString(e));
      resident = std::max(1, per_sm) * std::max(1, sms);
      g_resident_ctas[key] = resident;
    }
  }
  const unsigned grid = (unsigned)std::min<int64_t>(n_rows, resident);
  fn<<<grid, kFwdThreads, 0, s>>>(a);
  count_launches(1);
  return check_launch(who);
}

}  // namespace fastrl

extern "C" grpo_status grpo_logp_fwd(const void* logits, int32_t logits_dtype, int64_t row_stride,
                                     const int64_t* row_index, int64_t n_rows, int32_t V,
                                     const int32_t* y, float* logp_out, int32_t* status,
                                     grpo_stream_t stream) {
  GRPO_TRACE("grpo_logp_fwd");
  clear_error();
  return logp_rows("grpo_logp_fwd", logits, logits_dtype, row_stride, row_index, n_rows, nullptr,
                   V, y, logp_out, nullptr, status, as_stream(stream));
}

// ---- allocation-free variant ------------------------------------------------------------------
//
// Some callers cannot allocate device memory at the point where they run the loss: for
// example a plugin or custom-op host that hands over only input and output buffers and offers
// no workspace hook, or a runtime that forbids allocation after its start-up phase (to keep
// memory use fixed and latency predictable).  For them, grpo_loss_fwd_bwd_noalloc keeps the
// per-row loss scratch in a fixed array of this library instead of a caller workspace.
//
// The array below lives in every GPU that loads the library, until the process exits.  Host
// code cannot use its name as an address (on the host it names a stand-in object), so the
// device address is looked up with cudaGetSymbolAddress, once per device, with that device
// current, on the first call made on it.

namespace fastrl {
namespace {

constexpr int64_t kNoAllocMaxRows = 262144;  // 2 MiB of fp64 row-loss scratch
static __device__ __align__(256) double g_noalloc_row_loss[kNoAllocMaxRows];

constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kNoAllocMaxDevices] = {nullptr};

}  // namespace
}  // namespace fastrl

extern "C" grpo_status grpo_loss_fwd_bwd_noalloc(
    const void* logits, int32_t logits_dtype, int64_t row_stride, const int64_t* row_index,
    int64_t n_rows, int32_t V, const int32_t* y, const float* old_logp, const float* ref_logp,
    const float* adv, const int32_t* row_rollout, float eps_low, float eps_high, float beta,
    int32_t agg_mode, int64_t denom_tokens, const int64_t* seq_off, int64_t n_seq, void* dlogits,
    int32_t dlogits_dtype, float* logp_out, double* row_loss_out, double* loss_out, int32_t* status,
    grpo_stream_t stream) {
  GRPO_TRACE("grpo_loss_fwd_bwd_noalloc");
  clear_error();
  const char* who = "grpo_loss_fwd_bwd_noalloc";
  if (row_loss_out != nullptr)  // the caller's row-loss buffer is the only scratch: none needed
    return grpo_loss_fwd_bwd(logits, logits_dtype, row_stride, row_index, n_rows, V, y, old_logp,
                             ref_logp, adv, row_rollout, eps_low, eps_high, beta, agg_mode,
                             denom_tokens, seq_off, n_seq, dlogits, dlogits_dtype, logp_out,
                             row_loss_out, loss_out, status, nullptr, nullptr, stream);
  if (n_rows > kNoAllocMaxRows)
    return fail(GRPO_ERR_UNSUPPORTED,
                "%s: n_rows = %lld exceeds the fixed scratch of %lld rows; pass row_loss_out, "
                "split the rows into calls of at most %lld, or use grpo_loss_fwd_bwd",
                who, (long long)n_rows, (long long)kNoAllocMaxRows, (long long)kNoAllocMaxRows);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: cudaGetDevice: %s", who, cudaGetErrorString(e));
  if (dev < 0 || dev >= kNoAllocMaxDevices)
    return fail(GRPO_ERR_UNSUPPORTED, "%s: device %d beyond %d", who, dev, kNoAllocMaxDevices);
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (g_noalloc_ptr[dev] == nullptr) {
      e = cudaGetSymbolAddress(&g_noalloc_ptr[dev], g_noalloc_row_loss);
      if (e != cudaSuccess) {
        g_noalloc_ptr[dev] = nullptr;
        return fail(GRPO_ERR_CUDA, "%s: cudaGetSymbolAddress of the scratch array: %s", who,
                    cudaGetErrorString(e));
      }
    }
    scratch = g_noalloc_ptr[dev];
  }
  // Every row loss the sum reads is written by the same call, so the scratch needs no clearing.
  size_t bytes = sizeof(g_noalloc_row_loss);
  return grpo_loss_fwd_bwd(logits, logits_dtype, row_stride, row_index, n_rows, V, y, old_logp,
                           ref_logp, adv, row_rollout, eps_low, eps_high, beta, agg_mode,
                           denom_tokens, seq_off, n_seq, dlogits, dlogits_dtype, logp_out,
                           nullptr, loss_out, status, n_rows > 0 ? scratch : nullptr,
                           n_rows > 0 ? &bytes : nullptr, stream);
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_loss)
}  // namespace fastrl
