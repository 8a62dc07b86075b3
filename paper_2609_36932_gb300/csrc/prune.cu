// grpo_prune: maximising-differential advantage pruning (MDAP), Sec. 3.2 Eqs. 6-9, with the
// traversal order, per-class guarantee and DP-alignment fill of Algorithm 1 (Phase 2).
//
// Kernels, in stream order (0 first):
//   1. the n-gram sets N_n(o_i) of Eq. 7, one CTA per rollout:
//        n = 1   unigram_set_kernel: a bitmap over the vocabulary built in shared memory;
//        n = 2,3 ngram_set_kernel: each length-n window packed into a 64-bit key (18 bits per id),
//                bitonic-sorted (shared memory when it fits, else the workspace), repeats dropped;
//   2. the pair test theta_ij < tau for every pair i < j of a prompt with equal rewards:
//        n = 1   bitmap_pair_kernel: |N_i & N_j| = popcount of the AND, one CTA per pair;
//        n = 2,3 sorted_pair_kernel: binary search of the smaller set in the larger, a warp per pair;
//      each writes one byte per ordered pair: 1 when the two are in one class and too close;
//   0. class_kernel, one warp per prompt: advantage classes (exact reward equality, or chained
//      advantages for continuous rewards) and the fp64 |r - mean| visiting order;
//   3. select_kernel, one warp per prompt: the greedy of Eq. 8 as bitmask operations and the
//      per-prompt cap by round-robin over classes;
//   4. dp_fill_kernel (dp_divisor > 1), one thread: cyclic fill to a multiple of the divisor.
// For n = 1 with at most 64 KiB of bitmaps per prompt, prune_unigram_fused_kernel does steps 0-3
// in one CTA per prompt, in shared memory.
// Every decision is an integer or exactly rounded fp64 operation, so the keep mask is bit-exact.
#define GRPO_TU 1  // this file's bit in the checked build's report (grpo_debug_checks)
#include <algorithm>
#include <atomic>

#include "common.cuh"
#include "trace.cuh"

namespace fastrl {
namespace {

constexpr int kSortThreads = 512;
constexpr int kSmemKeys = 8192;  // keys sorted in shared memory (64 KiB); larger sets use ws
constexpr uint64_t kSentinel = ~0ull;  // sorts after every real key (< 2^54)
constexpr int kMaxG = 32;

struct PruneWs {
  uint64_t* keys;     // n >= 2: [2T]; rollout r owns keys[2*off[r] .. 2*off[r+1])
  uint64_t* bitmaps;  // n == 1: [P*G][words]
  int32_t* nuniq;     // [P*G] set sizes
  int32_t* cls;       // [P*G] class label: the smallest index in the rollout's class
  int32_t* rank;      // [P*G] visiting position inside the prompt
  uint8_t* close;     // [P*G*G]: close[(p*G + i)*G + j] = 1 if same class and theta_ij < tau
  int words;          // ceil(V / 64)
};

__host__ __device__ inline int bitmap_words(int V) { return (V + 63) / 64; }

size_t prune_ws_bytes(int64_t T, int P, int G, int V, int n) {
  const size_t keys = n >= 2 ? (size_t)(2 * T) * 8 : 0;
  const size_t bitmaps = n == 1 ? (size_t)P * G * bitmap_words(V) * 8 : 0;
  return align_up(keys, 256) + align_up(bitmaps, 256) + 3 * align_up((size_t)P * G * 4, 256) +
         align_up((size_t)P * G * G, 256);
}

PruneWs prune_ws(void* ws, int64_t T, int P, int G, int V, int n) {
  char* p = static_cast<char*>(ws);
  PruneWs w;
  w.words = bitmap_words(V);
  w.keys = reinterpret_cast<uint64_t*>(p);
  p += align_up(n >= 2 ? (size_t)(2 * T) * 8 : 0, 256);
  w.bitmaps = reinterpret_cast<uint64_t*>(p);
  p += align_up(n == 1 ? (size_t)P * G * w.words * 8 : 0, 256);
  w.nuniq = reinterpret_cast<int32_t*>(p);
  p += align_up((size_t)P * G * 4, 256);
  w.cls = reinterpret_cast<int32_t*>(p);
  p += align_up((size_t)P * G * 4, 256);
  w.rank = reinterpret_cast<int32_t*>(p);
  p += align_up((size_t)P * G * 4, 256);
  w.close = reinterpret_cast<uint8_t*>(p);
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
  // the keys fit their buffer: the launch's shared memory, or the rollout's 2L workspace keys
  if (!GRPO_DCHECK(arr == skeys ? (size_t)np2 * 8 <= dynamic_smem_bytes() : np2 <= 2 * L)) {
    if (threadIdx.x == 0) w.nuniq[r] = 0;
    return;
  }
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

// theta_ij < tau (Eqs. 7-8), from integer set sizes; two empty sets have theta = 0.
__device__ bool too_close(int I, int ni, int nj, float tau) {
  const int U = ni + nj - I;
  if (U == 0) return 0.0 < (double)tau;
  const double theta = __dsub_rn(1.0, __ddiv_rn((double)I, (double)U));
  return theta < (double)tau;
}

// pair index k of a prompt -> (i, j), i < j, in row-major order of the upper triangle
__device__ void pair_of(int k, int G, int& i, int& j) {
  i = 0;
  while (k >= G - 1 - i) {
    k -= G - 1 - i;
    ++i;
  }
  j = i + 1 + k;
}

__global__ void unigram_set_kernel(const int32_t* __restrict__ ids, const int64_t* __restrict__ off,
                                   int V, PruneWs w, int32_t* status) {
  extern __shared__ __align__(16) unsigned long long bm[];
  __shared__ int warp_cnt[32];
  const int r = blockIdx.x;
  const int64_t o = off[r];
  const int64_t L = off[r + 1] - o;
  if (!GRPO_DCHECK((size_t)w.words * 8 <= dynamic_smem_bytes() && blockDim.x <= 1024)) {
    if (threadIdx.x == 0) w.nuniq[r] = 0;
    return;
  }
  for (int k = threadIdx.x; k < w.words; k += blockDim.x) bm[k] = 0ull;
  __syncthreads();
  bool bad = false;
  for (int64_t t = threadIdx.x; t < L; t += blockDim.x) {
    const int32_t id = ids[o + t];
    if (id < 0 || id >= V) {
      bad = true;
      continue;
    }
    atomicOr(&bm[id >> 6], 1ull << (id & 63));
  }
  if (bad && status) atomicOr(status, GRPO_DEVFLAG_BAD_TOKEN);
  __syncthreads();
  uint64_t* out = w.bitmaps + (int64_t)r * w.words;
  int cnt = 0;
  for (int k = threadIdx.x; k < w.words; k += blockDim.x) {
    const unsigned long long v = bm[k];
    out[k] = v;
    cnt += __popcll(v);
  }
  for (int s = 16; s > 0; s >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, s);
  if ((threadIdx.x & 31) == 0) warp_cnt[threadIdx.x >> 5] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    int total = 0;
    for (int q = 0; q < (int)(blockDim.x >> 5); ++q) total += warp_cnt[q];
    w.nuniq[r] = total;
  }
}

constexpr int kPairThreads = 256;
constexpr int kPairUnroll = 4;

__global__ void __launch_bounds__(kPairThreads) bitmap_pair_kernel(int G, float tau, PruneWs w) {
  __shared__ int warp_cnt[32];
  const int pairs = G * (G - 1) / 2;
  const int p = blockIdx.x / pairs;
  int i, j;
  pair_of(blockIdx.x % pairs, G, i, j);
  const int ri = p * G + i, rj = p * G + j;
  uint8_t* close = w.close + (int64_t)p * G * G;
  if (w.cls[ri] != w.cls[rj]) {  // different classes never compare (Eq. 8 is per class)
    if (threadIdx.x == 0) close[i * G + j] = close[j * G + i] = 0;
    return;
  }
  const uint64_t* a = w.bitmaps + (int64_t)ri * w.words;
  const uint64_t* b = w.bitmaps + (int64_t)rj * w.words;
  int cnt = 0;
  // kPairUnroll independent loads of each bitmap per thread before any is used
  for (int k0 = threadIdx.x; k0 < w.words; k0 += blockDim.x * kPairUnroll) {
    uint64_t x[kPairUnroll], y[kPairUnroll];
#pragma unroll
    for (int u = 0; u < kPairUnroll; ++u) {
      const int k = k0 + u * (int)blockDim.x;
      x[u] = k < w.words ? a[k] : 0ull;
      y[u] = k < w.words ? b[k] : 0ull;
    }
#pragma unroll
    for (int u = 0; u < kPairUnroll; ++u) cnt += __popcll(x[u] & y[u]);
  }
  for (int s = 16; s > 0; s >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, s);
  if ((threadIdx.x & 31) == 0) warp_cnt[threadIdx.x >> 5] = cnt;
  __syncthreads();
  if (threadIdx.x == 0) {
    int I = 0;
    for (int q = 0; q < (int)(blockDim.x >> 5); ++q) I += warp_cnt[q];
    close[i * G + j] = close[j * G + i] = too_close(I, w.nuniq[ri], w.nuniq[rj], tau) ? 1 : 0;
  }
}

__global__ void sorted_pair_kernel(const int64_t* __restrict__ off, int P, int G, float tau,
                                   PruneWs w) {
  const int pairs = G * (G - 1) / 2;
  const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (int64_t)P * pairs) return;
  const int p = (int)(gw / pairs);
  int i, j;
  pair_of((int)(gw % pairs), G, i, j);
  const int ri = p * G + i, rj = p * G + j;
  uint8_t* close = w.close + (int64_t)p * G * G;
  if (w.cls[ri] != w.cls[rj]) {
    if (lane == 0) close[i * G + j] = close[j * G + i] = 0;
    return;
  }
  int na = w.nuniq[ri], nb = w.nuniq[rj];
  const uint64_t* a = w.keys + 2 * off[ri];
  const uint64_t* b = w.keys + 2 * off[rj];
  // each set lies in its rollout's 2L keys of the workspace
  if (!GRPO_DCHECK(na >= 0 && nb >= 0 && na <= 2 * (off[ri + 1] - off[ri]) &&
                   nb <= 2 * (off[rj + 1] - off[rj]))) {
    if (lane == 0) close[i * G + j] = close[j * G + i] = 0;
    return;
  }
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
  if (lane == 0)
    close[i * G + j] = close[j * G + i] = too_close(cnt, w.nuniq[ri], w.nuniq[rj], tau) ? 1 : 0;
}

// |r_i - mean| in fp64 with Eq. 5's index-order mean; the visiting key of Algorithm 1.
__device__ void group_dist(const float* r, int G, double* dist) {
  double sum = 0.0;
  for (int i = 0; i < G; ++i) sum = __dadd_rn(sum, (double)r[i]);
  const double mean = __ddiv_rn(sum, (double)G);
  for (int i = 0; i < G; ++i) dist[i] = fabs(__dsub_rn((double)r[i], mean));
}

// Classes and visiting order, one warp per prompt (lane i holds rollout i, G <= 32).
//   classes: exact reward equality (Eq. 6 for discrete rewards), or, with class_eps > 0, chains
//     of the advantages sorted ascending (ties by index) whose consecutive gaps are < class_eps
//     (the continuous-reward grouping |A_i - A_j| < eps, closed under transitivity);
//   visiting order: |A| descending as |r - mean| descending (fp64, Eq. 5's index-order mean),
//     lower index first on ties.
// One warp: advantage classes and visiting ranks of prompt p's rollouts, written to cls[0..G)
// and rank[0..G) (global workspace or shared memory).
__device__ void classify_warp(const float* __restrict__ rewards, const float* __restrict__ adv,
                              float class_eps, int p, int G, int lane, int32_t* cls, int32_t* rnk) {
  constexpr unsigned FULL = 0xffffffffu;
  const bool act = lane < G;
  const float r = act ? rewards[(int64_t)p * G + lane] : 0.f;
  double sum = 0.0;
  for (int i = 0; i < G; ++i) sum = __dadd_rn(sum, (double)__shfl_sync(FULL, r, i));
  const double mean = __ddiv_rn(sum, (double)G);
  const double dist = act ? fabs(__dsub_rn((double)r, mean)) : -1.0;
  int rank = 0;
  for (int j = 0; j < G; ++j) {
    const double dj = __shfl_sync(FULL, dist, j);
    rank += (dj > dist || (dj == dist && j < lane)) ? 1 : 0;
  }
  int label = lane;
  if (class_eps <= 0.f) {
    for (int j = G - 1; j >= 0; --j)  // smallest j with an equal reward
      if (__shfl_sync(FULL, r, j) == r) label = j;
  } else {
    const float a = act ? adv[(int64_t)p * G + lane] : 0.f;
    int spos = 0;  // position when sorted by a ascending, ties by index
    for (int j = 0; j < G; ++j) {
      const float aj = __shfl_sync(FULL, a, j);
      spos += (aj < a || (aj == a && j < lane)) ? 1 : 0;
    }
    float prev = a;
    for (int j = 0; j < G; ++j) {
      const float aj = __shfl_sync(FULL, a, j);
      const int sj = __shfl_sync(FULL, spos, j);
      if (sj == spos - 1) prev = aj;
    }
    const bool brk = act && (spos == 0 || __dsub_rn((double)a, (double)prev) >= (double)class_eps);
    int chain = 0;  // breaks at or before my sorted position
    for (int j = 0; j < G; ++j) {
      const int sj = __shfl_sync(FULL, spos, j);
      const bool bj = __shfl_sync(FULL, brk, j);
      chain += (bj && sj <= spos) ? 1 : 0;
    }
    for (int j = G - 1; j >= 0; --j)
      if (__shfl_sync(FULL, chain, j) == chain) label = j;
  }
  if (act) {
    cls[lane] = label;
    rnk[lane] = rank;
  }
}

__global__ void class_kernel(const float* __restrict__ rewards, const float* __restrict__ adv,
                             float class_eps, int P, int G, PruneWs w) {
  const int p = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (p >= P) return;  // uniform per warp
  classify_warp(rewards, adv, class_eps, p, G, threadIdx.x & 31, w.cls + (int64_t)p * G,
                w.rank + (int64_t)p * G);
}

// One warp per prompt: the greedy of Eq. 8 and the per-prompt cap as bitmask operations.
// One warp: the greedy of Eq. 8 and the per-prompt cap for one prompt, from its ranks, class
// labels and G x G closeness bytes; writes keep[0..G) and *kept.
__device__ void select_warp(int G, int keep_cap, const int32_t* rnk, const int32_t* cls_in,
                            const uint8_t* close, int lane, uint8_t* __restrict__ keep,
                            int32_t* __restrict__ kept_out) {
  constexpr unsigned FULL = 0xffffffffu;
  const bool act = lane < G;
  const int rank = act ? rnk[lane] : 64 + lane;
  const int label = act ? cls_in[lane] : -1 - lane;
  // same-class rollouts within tau of this one
  uint32_t near = 0;
  if (act) {
    const uint8_t* row = close + lane * G;
    for (int j = 0; j < G; ++j)
      if (j != lane && row[j]) near |= 1u << j;
  }
  // Eq. 8, greedily along the visiting order
  uint32_t kept = 0;
  for (int a = 0; a < G; ++a) {
    const int i = __ffs(__ballot_sync(FULL, act && rank == a)) - 1;
    if (!GRPO_DCHECK(i >= 0 && i < G)) continue;  // the ranks are a permutation of 0..G-1
    if ((__shfl_sync(FULL, near, i) & kept) == 0) kept |= 1u << i;
  }
  int count = __popc(kept);
  // Per-prompt cap: classes take turns in visiting order of their first member; each turn adds
  // the class's next kept member in visiting order.  Equivalently keep the keep_cap kept
  // rollouts with the smallest (turn, class position).
  if (count > keep_cap) {
    const bool mine = act && ((kept >> lane) & 1u);
    uint32_t cls = 0;  // kept rollouts of my class
    for (int i = 0; i < G; ++i) {
      const int li = __shfl_sync(FULL, label, i);
      const uint32_t m = __ballot_sync(FULL, act && ((kept >> lane) & 1u) && label == li);
      if (lane == i) cls = m;
    }
    int turn = 0, crank = 64;
    for (int j = 0; j < G; ++j) {
      const int rj = __shfl_sync(FULL, rank, j);
      if ((cls >> j) & 1u) {
        turn += rj < rank ? 1 : 0;
        crank = min(crank, rj);
      }
    }
    const int key = turn * 64 + crank;
    int before = 0;
    for (int j = 0; j < G; ++j) {
      const int kj = __shfl_sync(FULL, key, j);
      before += (((kept >> j) & 1u) && kj < key) ? 1 : 0;
    }
    kept = __ballot_sync(FULL, mine && before < keep_cap);
    count = keep_cap;
  }
  if (act) keep[lane] = (kept >> lane) & 1u;
  if (lane == 0) *kept_out = count;
}

__global__ void select_kernel(int P, int G, int keep_cap, PruneWs w, uint8_t* __restrict__ keep,
                              int32_t* __restrict__ kept_per_prompt) {
  const int p = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (p >= P) return;  // uniform per warp
  select_warp(G, keep_cap, w.rank + (int64_t)p * G, w.cls + (int64_t)p * G,
              w.close + (int64_t)p * G * G, threadIdx.x & 31, keep + (int64_t)p * G,
              kept_per_prompt + p);
}

// n = 1 with small vocabulary bitmaps: the four steps above in one CTA per prompt (classes and
// ranks, bitmaps and set sizes, pair tests, selection), with every intermediate in shared
// memory.  Same arithmetic and decisions as the separate kernels.  Measured on GB300: it saves
// launches where each prompt's work is small (V = 1024: 26 us against 30 us for the selection),
// ties at V = 32000, and loses at V = 152064 (one CTA per prompt is too little parallelism for
// 8 x 19 KiB bitmaps and 28 pair tests), so it is used up to 64 KiB of bitmaps per prompt.
constexpr int kFusedThreads = 1024;
constexpr size_t kFusedMaxBitmapBytes = 64 * 1024;

__global__ void __launch_bounds__(kFusedThreads)
    prune_unigram_fused_kernel(const float* __restrict__ rewards, const float* __restrict__ adv,
                               float class_eps, const int32_t* __restrict__ ids,
                               const int64_t* __restrict__ off, int G, int V, int words, float tau,
                               int keep_cap, uint8_t* __restrict__ keep,
                               int32_t* __restrict__ kept_per_prompt, int32_t* status) {
  extern __shared__ __align__(16) unsigned long long bms[];  // [G][words]
  __shared__ int32_t s_cls[kMaxG], s_rank[kMaxG], s_nuniq[kMaxG];
  __shared__ uint8_t s_close[kMaxG * kMaxG];
  __shared__ int64_t s_off[kMaxG + 1];
  const int p = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarps = kFusedThreads / 32;
  if (!GRPO_DCHECK(G <= kMaxG && (size_t)G * words * 8 <= dynamic_smem_bytes())) return;
  if (warp == 0) classify_warp(rewards, adv, class_eps, p, G, lane, s_cls, s_rank);
  if (tid <= G) s_off[tid] = off[(int64_t)p * G + tid];
  for (int k = tid; k < G * words; k += kFusedThreads) bms[k] = 0ull;
  __syncthreads();
  // all tokens of the prompt in one flat loop (independent loads); a token's rollout is the
  // last r with s_off[r] <= its index
  bool bad = false;
  const int64_t t0 = s_off[0], t1 = s_off[G];
  for (int64_t t = t0 + tid; t < t1; t += kFusedThreads) {
    const int32_t id = ids[t];
    int r = 0;
    while (r + 1 < G && s_off[r + 1] <= t) ++r;
    if (id < 0 || id >= V) {
      bad = true;
      continue;
    }
    atomicOr(&bms[(int64_t)r * words + (id >> 6)], 1ull << (id & 63));
  }
  if (bad && status) atomicOr(status, GRPO_DEVFLAG_BAD_TOKEN);
  __syncthreads();
  for (int r = warp; r < G; r += kWarps) {  // |N_r|
    int c = 0;
    for (int k = lane; k < words; k += 32) c += __popcll(bms[(int64_t)r * words + k]);
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (lane == 0) s_nuniq[r] = c;
  }
  __syncthreads();
  const int pairs = G * (G - 1) / 2;
  for (int q = warp; q < pairs; q += kWarps) {  // theta_ij < tau for same-class pairs
    int i, j;
    pair_of(q, G, i, j);
    uint8_t c = 0;
    if (s_cls[i] == s_cls[j]) {
      const unsigned long long* a = bms + (int64_t)i * words;
      const unsigned long long* b = bms + (int64_t)j * words;
      int I = 0;
      for (int k = lane; k < words; k += 32) I += __popcll(a[k] & b[k]);
      for (int o = 16; o > 0; o >>= 1) I += __shfl_xor_sync(0xffffffffu, I, o);
      c = too_close(I, s_nuniq[i], s_nuniq[j], tau) ? 1 : 0;
    }
    if (lane == 0) s_close[i * G + j] = s_close[j * G + i] = c;
  }
  __syncthreads();
  if (warp == 0)
    select_warp(G, keep_cap, s_rank, s_cls, s_close, lane, keep + (int64_t)p * G,
                kept_per_prompt + p);
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

extern "C" grpo_status grpo_prune(const float* rewards, const float* adv, float class_eps,
                                  const int32_t* ids, const int64_t* off, int32_t P, int32_t G,
                                  int64_t T, int32_t V, int32_t ngram_n, float tau, int32_t keep_cap,
                                  int32_t dp_divisor, uint8_t* keep, int32_t* kept_per_prompt,
                                  int32_t* status, void* ws, size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_prune");
  clear_error();
  if (!(class_eps >= 0.f)) return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: class_eps must be >= 0");
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
  const grpo_status ws_ok =
      workspace_check(ws, ws_bytes, prune_ws_bytes(T, P, G, V, ngram_n), "grpo_prune", &query);
  if (ws_ok != GRPO_OK || query) return ws_ok;
  if (P == 0) return GRPO_OK;
  if (!rewards || !off || !keep || !kept_per_prompt || (T > 0 && !ids) || (class_eps > 0.f && !adv))
    return fail(GRPO_ERR_INVALID_ARG, "grpo_prune: NULL array");
  cudaStream_t s = as_stream(stream);
  const PruneWs w = prune_ws(ws, T, P, G, V, ngram_n);
  const int nroll = P * G;
  const int pairs = G * (G - 1) / 2;
  const unsigned warp_blocks = (unsigned)(((int64_t)P * 32 + 127) / 128);
  int launches = 0;
  const size_t fused_smem = (size_t)G * w.words * 8;
  if (ngram_n == 1 && fused_smem <= kFusedMaxBitmapBytes) {
    static std::atomic<uint64_t> fused_attr{0};  // bit d: the attribute is set on device d
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = dev < 64 ? (1ull << dev) : 0ull;
    if (!bit || !(fused_attr.load() & bit)) {  // once per device, before any stream capture
      if (cudaFuncSetAttribute(prune_unigram_fused_kernel,
                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)kFusedMaxBitmapBytes) != cudaSuccess)
        return check_launch("grpo_prune: cudaFuncSetAttribute");
      fused_attr.fetch_or(bit);
    }
    prune_unigram_fused_kernel<<<P, kFusedThreads, fused_smem, s>>>(
        rewards, adv, class_eps, ids, off, G, V, w.words, tau, keep_cap, keep, kept_per_prompt,
        status);
    launches = 1;
    if (dp_divisor > 1) {
      dp_fill_kernel<<<1, 32, 0, s>>>(rewards, P, G, dp_divisor, keep, kept_per_prompt);
      ++launches;
    }
    count_launches(launches);
    return check_launch("grpo_prune");
  }
  class_kernel<<<warp_blocks, 128, 0, s>>>(rewards, adv, class_eps, P, G, w);
  launches = 1;
  if (ngram_n == 1) {
    unigram_set_kernel<<<nroll, 256, (size_t)w.words * 8, s>>>(ids, off, V, w, status);
    ++launches;
    if (pairs > 0) {
      bitmap_pair_kernel<<<(unsigned)((int64_t)P * pairs), kPairThreads, 0, s>>>(G, tau, w);
      ++launches;
    }
  } else {
    const int smem = kSmemKeys * 8;
    static std::atomic<uint64_t> attr_set{0};  // bit d: the attribute is set on device d
    int dev = 0;
    cudaGetDevice(&dev);
    const uint64_t bit = dev < 64 ? (1ull << dev) : 0ull;
    if (!bit || !(attr_set.load() & bit)) {  // once per device, before any stream capture
      if (cudaFuncSetAttribute(ngram_set_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
          cudaSuccess)
        return check_launch("grpo_prune: cudaFuncSetAttribute");
      attr_set.fetch_or(bit);
    }
    ngram_set_kernel<<<nroll, kSortThreads, smem, s>>>(ids, off, V, ngram_n, w, status);
    ++launches;
    if (pairs > 0) {
      const int tpb = 256;
      const int64_t blocks = ((int64_t)P * pairs * 32 + tpb - 1) / tpb;
      sorted_pair_kernel<<<(unsigned)blocks, tpb, 0, s>>>(off, P, G, tau, w);
      ++launches;
    }
  }
  select_kernel<<<warp_blocks, 128, 0, s>>>(P, G, keep_cap, w, keep, kept_per_prompt);
  ++launches;
  if (dp_divisor > 1) {
    dp_fill_kernel<<<1, 32, 0, s>>>(rewards, P, G, dp_divisor, keep, kept_per_prompt);
    ++launches;
  }
  count_launches(launches);
  return check_launch("grpo_prune");
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_prune)
}  // namespace fastrl
