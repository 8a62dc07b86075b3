// grpo_compact: compaction of the kept rollouts' tokens.  Sec. 3.2 (after Eq. 9) feeds only the
// retained trajectories to the models, so the loss runs over their tokens only.
//
//   compact_scan_kernel  one CTA: exclusive scan of (kept, kept length) over the rollouts in
//                        tiles of the CTA width -> kept_idx, kept_off, counts {K, T_kept}.
//   compact_fill_kernel  one CTA per rollout: a kept rollout finds its position k by binary
//                        search in kept_idx and writes its token indices and rollout id.
#define GRPO_TU 2  // this file's bit in the checked build's report (grpo_debug_checks)
#include "common.cuh"
#include "trace.cuh"

namespace fastrl {
namespace {

constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads)
    compact_scan_kernel(const uint8_t* __restrict__ keep, const int64_t* __restrict__ off, int n,
                        int32_t* __restrict__ kept_idx, int64_t* __restrict__ kept_off,
                        int64_t* __restrict__ counts) {
  __shared__ int wk[kScanThreads / 32];
  __shared__ int64_t wt[kScanThreads / 32];
  __shared__ int carry_k;
  __shared__ int64_t carry_t;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    carry_k = 0;
    carry_t = 0;
  }
  __syncthreads();
  for (int base = 0; base < n; base += kScanThreads) {
    const int r = base + threadIdx.x;
    const bool kept = r < n && keep[r] != 0;
    const int64_t len = kept ? off[r + 1] - off[r] : 0;
    // inclusive scans inside the warp
    int ck = kept ? 1 : 0;
    int64_t ct = len;
    for (int s = 1; s < 32; s <<= 1) {
      const int ok = __shfl_up_sync(0xffffffffu, ck, s);
      const int64_t ot = __shfl_up_sync(0xffffffffu, ct, s);
      if (lane >= s) {
        ck += ok;
        ct += ot;
      }
    }
    if (lane == 31) {
      wk[warp] = ck;
      wt[warp] = ct;
    }
    __syncthreads();
    if (threadIdx.x == 0) {  // warp totals -> exclusive warp offsets (fixed order)
      int ak = 0;
      int64_t at = 0;
      for (int w = 0; w < kScanThreads / 32; ++w) {
        const int k = wk[w];
        const int64_t t = wt[w];
        wk[w] = ak;
        wt[w] = at;
        ak += k;
        at += t;
      }
    }
    __syncthreads();
    if (kept) {
      const int k = carry_k + wk[warp] + ck - 1;
      if (GRPO_DCHECK(k >= 0 && k <= r)) {  // k kept rollouts precede r
        kept_idx[k] = r;
        kept_off[k] = carry_t + wt[warp] + ct - len;
      }
    }
    __syncthreads();
    if (threadIdx.x == kScanThreads - 1) {  // last thread holds the tile totals
      carry_k += wk[warp] + ck;
      carry_t += wt[warp] + ct;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    kept_off[carry_k] = carry_t;
    counts[0] = carry_k;
    counts[1] = carry_t;
  }
}

__global__ void compact_fill_kernel(const uint8_t* __restrict__ keep, const int64_t* __restrict__ off,
                                    const int32_t* __restrict__ kept_idx,
                                    const int64_t* __restrict__ kept_off,
                                    const int64_t* __restrict__ counts,
                                    int64_t* __restrict__ src_token,
                                    int32_t* __restrict__ token_rollout) {
  const int r = blockIdx.x;
  if (!keep[r]) return;
  int lo = 0, hi = (int)counts[0];  // first k with kept_idx[k] >= r
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (kept_idx[mid] < r)
      lo = mid + 1;
    else
      hi = mid;
  }
  // the search found r, and its tokens end within the kept total
  if (!GRPO_DCHECK(lo < (int)counts[0] && kept_idx[lo] == r)) return;
  const int64_t dst = kept_off[lo];
  const int64_t o = off[r], L = off[r + 1] - o;
  if (!GRPO_DCHECK(dst >= 0 && dst + L <= counts[1])) return;
  for (int64_t s = threadIdx.x; s < L; s += blockDim.x) {
    src_token[dst + s] = o + s;
    token_rollout[dst + s] = r;
  }
}

}  // namespace
}  // namespace fastrl

using namespace fastrl;

extern "C" grpo_status grpo_compact(const uint8_t* keep, const int64_t* off, int32_t n_rollouts,
                                    int32_t* kept_idx, int64_t* kept_off, int64_t* src_token,
                                    int32_t* token_rollout, int64_t* counts, int64_t* counts_host,
                                    grpo_stream_t stream) {
  GRPO_TRACE("grpo_compact");
  clear_error();
  if (n_rollouts < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_compact: n_rollouts < 0");
  if (!off || !kept_off || !counts || (n_rollouts > 0 && (!keep || !kept_idx)))
    return fail(GRPO_ERR_INVALID_ARG, "grpo_compact: NULL array");
  if (n_rollouts > 0 && (!src_token || !token_rollout))
    return fail(GRPO_ERR_INVALID_ARG, "grpo_compact: NULL token arrays");
  cudaStream_t s = as_stream(stream);
  compact_scan_kernel<<<1, kScanThreads, 0, s>>>(keep, off, n_rollouts, kept_idx, kept_off, counts);
  int launches = 1;
  if (n_rollouts > 0) {
    compact_fill_kernel<<<n_rollouts, 256, 0, s>>>(keep, off, kept_idx, kept_off, counts, src_token,
                                                    token_rollout);
    ++launches;
  }
  count_launches(launches);
  grpo_status st = check_launch("grpo_compact");
  if (st != GRPO_OK) return st;
  if (counts_host) {
    const cudaError_t e =
        cudaMemcpyAsync(counts_host, counts, 2 * sizeof(int64_t), cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess)
      return fail(GRPO_ERR_CUDA, "grpo_compact: copy of counts: %s", cudaGetErrorString(e));
  }
  return GRPO_OK;
}

extern "C" grpo_status grpo_upload_kept(const void* src_host, void* dst_dev, int64_t row_bytes,
                                        const uint8_t* keep_host, const int64_t* off_host,
                                        int32_t n_rollouts, int64_t* bytes_out,
                                        int32_t* copies_out, grpo_stream_t stream) {
  GRPO_TRACE("grpo_upload_kept");
  clear_error();
  if (bytes_out) *bytes_out = 0;
  if (copies_out) *copies_out = 0;
  if (n_rollouts < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_upload_kept: n_rollouts < 0");
  if (row_bytes <= 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_upload_kept: row_bytes <= 0");
  if (n_rollouts == 0) return GRPO_OK;
  if (!src_host || !dst_dev || !keep_host || !off_host)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_upload_kept: NULL array");
  if (off_host[0] < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_upload_kept: off_host[0] < 0");
  for (int32_t r = 0; r < n_rollouts; ++r)
    if (off_host[r + 1] < off_host[r])
      return fail(GRPO_ERR_INVALID_ARG, "grpo_upload_kept: off_host decreases at %d", r);
  if (off_host[n_rollouts] > INT64_MAX / row_bytes)
    return fail(GRPO_ERR_INVALID_ARG, "grpo_upload_kept: byte offsets overflow int64");
  cudaStream_t s = as_stream(stream);
  const char* src = static_cast<const char*>(src_host);
  char* dst = static_cast<char*>(dst_dev);
  int64_t bytes = 0;
  int32_t copies = 0;
  for (int32_t r = 0; r < n_rollouts;) {
    if (!keep_host[r]) {
      ++r;
      continue;
    }
    int32_t e = r;
    while (e < n_rollouts && keep_host[e]) ++e;  // kept run r..e-1
    const int64_t b0 = off_host[r] * row_bytes, n = (off_host[e] - off_host[r]) * row_bytes;
    if (n > 0) {
      const cudaError_t err =
          cudaMemcpyAsync(dst + b0, src + b0, (size_t)n, cudaMemcpyHostToDevice, s);
      if (err != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "grpo_upload_kept: copy of rollouts %d..%d: %s", r, e - 1,
                    cudaGetErrorString(err));
      bytes += n;
      ++copies;
      if (bytes_out) *bytes_out = bytes;
      if (copies_out) *copies_out = copies;
    }
    r = e;
  }
  return GRPO_OK;
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_compact)
}  // namespace fastrl
