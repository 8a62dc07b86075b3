// grpo_prune: maximising-differential advantage pruning (MDAP), Sec. 3.2 Eqs. 6-9, with the
// traversal order, per-class guarantee and DP-alignment fill of Algorithm 1 (Phase 2).
//
// Three kernels (a fourth when dp_divisor > 1):
//   1. ngram_set_kernel   one CTA per rollout: pack each length-n window of token ids into a
//                         64-bit key (18 bits per id), bitonic-sort the keys (in shared memory
//                         when they fit, else in the workspace), drop repeats -> N_n(o_i) (Eq. 7)
//                         as a sorted array plus its size.
//   2. intersect_kernel   one warp per pair (i < j) of a prompt with equal rewards: |N_i & N_j|
//                         by binary search of the smaller set's keys in the larger one.
//   3. select_kernel      one thread per prompt: fp64 |r - mean| order, greedy Eq. 8 per reward
//                         class, per-prompt cap by round-robin over classes.
//   4. dp_fill_kernel     one thread: cyclic fill until the kept total is a multiple of d.
// All decisions are integer or exactly rounded fp64 operations, so the keep mask is bit-exact.
#include <algorithm>

#include "common.cuh"

namespace fastrl {
namespace {

constexpr int kSortThreads = 512;
constexpr int kSmemKeys = 8192;  // keys sorted in shared memory (64 KiB); larger sets use ws
constexpr uint64_t kSentinel = ~0ull;  // sorts after every real key (< 2^54)
constexpr int kMaxG = 32;

struct PruneWs {
  uint64_t* keys;  // [2T]: rollout r owns keys[2*off[r] .. 2*off[r+1])
  int32_t* nuniq;  // [P*G]
  int32_t* inter;  // [P*G*G]
};

__host__ __device__ inline size_t ws_keys_bytes(int64_t T) { return (size_t)(2 * T) * 8; }

size_t prune_ws_bytes(int64_t T, int P, int G) {
  return align_up(ws_keys_bytes(T), 256) + align_up((size_t)P * G * 4, 256) +
         align_up((size_t)P * G * G * 4, 256);
}

PruneWs prune_ws(void* ws, int64_t T, int P, int G) {
  char* p = static_cast<char*>(ws);
  PruneWs w;
  w.keys = reinterpret_cast<uint64_t*>(p);
  p += align_up(ws_keys_bytes(T), 256);
  w.nuniq = reinterpret_cast<int32_t*>(p);
  p += align_up((size_t)P * G * 4, 256);
  w.inter = reinterpret_cast<int32_t*>(p);
  return w;
}

// Bitonic sort of arr[0..n), n a power of two, by one CTA.  Works on shared or global memory:
// __syncthreads orders a CTA's accesses to both.
__device__ void bitonic_sort(uint64_t* arr, int n) {
  for (int k = 2; k <= n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const uint64_t a = arr[i], b = arr[ixj];
          const bool ascending = (i & k) == 0;
          if ((a > b) == ascending) {
            arr[i] = b;
            arr[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
}

// Exclusive scan of one flag per thread over the CTA; returns the prefix, writes the total.
__device__ int block_exclusive_count(bool flag, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) warp_tot[warp] = __popc(bal);
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int w = 0; w < nw; ++w) {
      const int t = warp_tot[w];
      warp_tot[w] = acc;
      acc += t;
    }
    *total = acc;
  }
  __syncthreads();
  const int r = warp_tot[warp] + in_warp;
  return r;
}

__global__ void __launch_bounds__(kSortThreads)
    ngram_set_kernel(const int32_t* __restrict__ ids, const int64_t* __restrict__ off, int V,
                     int n, PruneWs w, int32_t* status) {
  extern __shared__ __align__(16) uint64_t skeys[];
  __shared__ int warp_tot[kSortThreads / 32];
  __shared__ int chunk_total;
  __shared__ uint64_t prev_last;
  __shared__ int out_base;
  const int r = blockIdx.x;
  const int64_t o = off[r];
  const int64_t L = off[r + 1] - o;
  const int c = L >= n ? (int)(L - n + 1) : 0;  // number of windows
  uint64_t* region = w.keys + 2 * o;            // room for 2L >= next power of two of c keys
  if (c == 0) {
    if (threadIdx.x == 0) w.nuniq[r] = 0;
    return;
  }
  int np2 = 1;
  while (np2 < c) np2 <<= 1;
  uint64_t* arr = np2 <= kSmemKeys ? skeys : region;
  bool bad = false;
  for (int k = threadIdx.x; k < np2; k += blockDim.x) {
    uint64_t key = kSentinel;
    if (k < c) {
      key = 0;
      for (int q = 0; q < n; ++q) {
        const int32_t id = ids[o + k + q];
        bad |= (id < 0 || id >= V);
        key |= (uint64_t)((uint32_t)id & 0x3FFFFu) << (18 * q);
      }
    }
    arr[k] = key;
  }
  if (bad && status) atomicOr(status, GRPO_DEVFLAG_BAD_TOKEN);
  __syncthreads();
  bitonic_sort(arr, np2);
  // Keep the first key of each run of equal keys, in order, at region[0 .. u).
  if (threadIdx.x == 0) out_base = 0;
  __syncthreads();
  for (int start = 0; start < c; start += blockDim.x) {
    const int i = start + threadIdx.x;
    uint64_t key = 0, before = 0;
    if (i < c) {
      key = arr[i];
      before = (i == 0) ? ~key : (threadIdx.x == 0 ? prev_last : arr[i - 1]);
    }
    const bool first = i < c && key != before;
    __syncthreads();  // every read of this chunk happens before any write below
    const int pos = block_exclusive_count(first, warp_tot, &chunk_total);
    if (first) region[out_base + pos] = key;
    const int last = min(c, start + (int)blockDim.x) - 1;
    if (i == last) prev_last = key;
    __syncthreads();
    if (threadIdx.x == 0) out_base += chunk_total;
    __syncthreads();
  }
  if (threadIdx.x == 0) w.nuniq[r] = out_base;
}

__global__ void intersect_kernel(const float* __restrict__ rewards, const int64_t* __restrict__ off,
                                 int P, int G, PruneWs w) {
  const int pairs_per_prompt = G * (G - 1) / 2;
  const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (int64_t)P * pairs_per_prompt) return;
  const int p = (int)(gw / pairs_per_prompt);
  int k = (int)(gw % pairs_per_prompt);
  int i = 0;
  while (k >= G - 1 - i) {  // pair index -> (i, j), i < j
    k -= G - 1 - i;
    ++i;
  }
  const int j = i + 1 + k;
  const int ri = p * G + i, rj = p * G + j;
  int32_t* inter = w.inter + (int64_t)p * G * G;
  if (rewards[ri] != rewards[rj]) {  // different classes never compare (Eq. 8 is per class)
    if (lane == 0) inter[i * G + j] = inter[j * G + i] = -1;
    return;
  }
  int na = w.nuniq[ri], nb = w.nuniq[rj];
  const uint64_t* a = w.keys + 2 * off[ri];
  const uint64_t* b = w.keys + 2 * off[rj];
  if (na > nb) {
    const uint64_t* t = a;
    a = b;
    b = t;
    const int tn = na;
    na = nb;
    nb = tn;
  }
  int cnt = 0;
  for (int e = lane; e < na; e += 32) {
    const uint64_t key = a[e];
    int lo = 0, hi = nb;  // first index with b[idx] >= key
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (b[mid] < key)
        lo = mid + 1;
      else
        hi = mid;
    }
    cnt += (lo < nb && b[lo] == key) ? 1 : 0;
  }
  for (int s = 16; s > 0; s >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, s);
  if (lane == 0) inter[i * G + j] = inter[j * G + i] = cnt;
}

// |r_i - mean| in fp64 with Eq. 5's index-order mean; the visiting key of Algorithm 1.
__device__ void group_dist(const float* r, int G, double* dist) {
  double sum = 0.0;
  for (int i = 0; i < G; ++i) sum = __dadd_rn(sum, (double)r[i]);
  const double mean = __ddiv_rn(sum, (double)G);
  for (int i = 0; i < G; ++i) dist[i] = fabs(__dsub_rn((double)r[i], mean));
}

// theta_ij < tau (Eqs. 7-8), from integer set sizes; two empty sets have theta = 0.
__device__ bool too_close(int I, int ni, int nj, float tau) {
  const int U = ni + nj - I;
  if (U == 0) return 0.0 < (double)tau;
  const double theta = __dsub_rn(1.0, __ddiv_rn((double)I, (double)U));
  return theta < (double)tau;
}

__global__ void select_kernel(const float* __restrict__ rewards, int P, int G, float tau,
                              int keep_cap, PruneWs w, uint8_t* __restrict__ keep,
                              int32_t* __restrict__ kept_per_prompt) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= P) return;
  const float* r = rewards + (int64_t)p * G;
  const int32_t* nu = w.nuniq + (int64_t)p * G;
  const int32_t* inter = w.inter + (int64_t)p * G * G;
  double dist[kMaxG];
  int order[kMaxG];
  bool kept[kMaxG];
  group_dist(r, G, dist);
  for (int i = 0; i < G; ++i) {  // stable insertion sort: dist descending, index ascending
    int k = i;
    while (k > 0 && dist[order[k - 1]] < dist[i]) {
      order[k] = order[k - 1];
      --k;
    }
    order[k] = i;
    kept[i] = false;
  }
  // Eq. 8, greedily along the visiting order, inside each reward class.
  int count = 0;
  for (int a = 0; a < G; ++a) {
    const int i = order[a];
    bool drop = false;
    for (int b = 0; b < a && !drop; ++b) {
      const int j = order[b];
      if (!kept[j] || r[j] != r[i]) continue;
      drop = too_close(inter[i * G + j], nu[i], nu[j], tau);
    }
    kept[i] = !drop;
    count += kept[i] ? 1 : 0;
  }
  // Per-prompt cap: classes (dist descending, then lowest member) take turns, each turn adding
  // its next kept member in index order.
  if (count > keep_cap) {
    int cls_first[kMaxG];  // class representative (its lowest index), in turn order
    int ncls = 0;
    for (int a = 0; a < G; ++a) {  // visiting order lists classes by (dist desc, first index)
      const int i = order[a];
      if (!kept[i]) continue;
      bool seen = false;
      for (int c = 0; c < ncls; ++c) seen |= (r[cls_first[c]] == r[i]);
      if (!seen) cls_first[ncls++] = i;
    }
    bool capped[kMaxG];
    int next[kMaxG];  // per class: next index to look at
    for (int i = 0; i < G; ++i) capped[i] = false;
    for (int c = 0; c < ncls; ++c) next[c] = 0;
    int taken = 0;
    while (taken < keep_cap) {
      for (int c = 0; c < ncls && taken < keep_cap; ++c) {
        const float rc = r[cls_first[c]];
        int i = next[c];
        while (i < G && !(kept[i] && r[i] == rc)) ++i;
        if (i < G) {
          capped[i] = true;
          ++taken;
          next[c] = i + 1;
        } else {
          next[c] = G;
        }
      }
    }
    for (int i = 0; i < G; ++i) kept[i] = capped[i];
    count = keep_cap;
  }
  for (int i = 0; i < G; ++i) keep[(int64_t)p * G + i] = kept[i] ? 1 : 0;
  kept_per_prompt[p] = count;
}

__global__ void dp_fill_kernel(const float* __restrict__ rewards, int P, int G, int d,
                               uint8_t* __restrict__ keep, int32_t* __restrict__ kept_per_prompt) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  int64_t total = 0;
  for (int p = 0; p < P; ++p) total += kept_per_prompt[p];
  int cursor = 0;
  double dist[kMaxG];
  while (total % d != 0) {
    bool added = false;
    for (int tries = 0; tries < P && !added; ++tries) {
      const int p = cursor;
      cursor = (cursor + 1) % P;
      group_dist(rewards + (int64_t)p * G, G, dist);
      int best = -1;
      for (int i = 0; i < G; ++i) {
        if (keep[(int64_t)p * G + i]) continue;
        if (best < 0 || dist[i] > dist[best]) best = i;
      }
      if (best >= 0) {
        keep[(int64_t)p * G + best] = 1;
        kept_per_prompt[p] += 1;
        ++total;
        added = true;
      }
    }
    if (!added) break;
  }
}

}  // namespace
}  // namespace fastrl

using namespace fastrl;

extern "C" grpo_status grpo_prune(const float* rewards, const int32_t* ids, const int64_t* off,
                                  int32_t P, int32_t G, int64_t T, int32_t V, int32_t ngram_n,
                                  float tau, int32_t keep_cap, int32_t dp_divisor, uint8_t* keep,
                                  int32_t* kept_per_prompt, int32_t* status, void* ws,
                                  size_t* ws_bytes, grpo_stream_t stream) {
  clear_error();
  if (P < 0 || T < 0) return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: P = %d, T = %lld", P, (long long)T);
  if (G < 1 || G > kMaxG) return fail(GRPO_ERR_UNSUPPORTED, "grpo_prune: G = %d not in [1, %d]", G, kMaxG);
  if (V < 1 || V > (1 << 18))
    return fail(GRPO_ERR_UNSUPPORTED, "grpo_prune: V = %d not in [1, 2^18]", V);
  if (ngram_n < 1 || ngram_n > 3)
    return fail(GRPO_ERR_UNSUPPORTED, "grpo_prune: ngram_n = %d not in [1, 3]", ngram_n);
  if (keep_cap < 1) return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: keep_cap = %d < 1", keep_cap);
  if (dp_divisor < 1) return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: dp_divisor = %d < 1", dp_divisor);
  if (tau != tau) return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: tau is NaN");
  bool query = false;
  const grpo_status ws_ok = workspace_check(ws, ws_bytes, prune_ws_bytes(T, P, G), "grpo_prune", &query);
  if (ws_ok != GRPO_OK || query) return ws_ok;
  if (P == 0) return GRPO_OK;
  if (!rewards || !off || !keep || !kept_per_prompt || (T > 0 && !ids))
    return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: NULL array");
  cudaStream_t s = as_stream(stream);
  const PruneWs w = prune_ws(ws, T, P, G);
  const int nroll = P * G;
  const int smem = kSmemKeys * 8;
  if (cudaFuncSetAttribute(ngram_set_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess)
    return check_launch("grpo_prune: cudaFuncSetAttribute");
  ngram_set_kernel<<<nroll, kSortThreads, smem, s>>>(ids, off, V, ngram_n, w, status);
  int launches = 1;
  const int64_t warps = (int64_t)P * (G * (G - 1) / 2);
  if (warps > 0) {
    const int tpb = 256;
    const int64_t blocks = (warps * 32 + tpb - 1) / tpb;
    intersect_kernel<<<(unsigned)blocks, tpb, 0, s>>>(rewards, off, P, G, w);
    ++launches;
  }
  select_kernel<<<(P + 127) / 128, 128, 0, s>>>(rewards, P, G, tau, keep_cap, w, keep, kept_per_prompt);
  ++launches;
  if (dp_divisor > 1) {
    dp_fill_kernel<<<1, 32, 0, s>>>(rewards, P, G, dp_divisor, keep, kept_per_prompt);
    ++launches;
  }
  count_launches(launches);
  return check_launch("grpo_prune");
}
