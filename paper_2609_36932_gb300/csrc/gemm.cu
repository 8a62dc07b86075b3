// The two products of the output layer's backward, on the tensor cores.  The chain rule through
// z = h W^T (the output layer whose logits Eqs. 1-3 consume, Sec. 3.2) turns the rows' dlogits
// into the gradients of the hidden states and of the weight:
//   dh = dlogits * W       C[t, d] = sum_v dl[t, v] W[v, d]    A = dl  (K-major: v contiguous)
//   dW = dlogits^T * h     C[v, d] = sum_t dl[t, v] h[t, d]    A = dl^T (M-major: v contiguous)
// In both, B (W or h) is stored [K][N] with N = d contiguous (N-major).  One kernel serves both:
//
//   C[M, N] (+)= sum_k A(m, k) B(k, n),  bf16 operands, f32 accumulation, f32 or bf16 C.
//
// A unit is a 256 x 256 tile of C (two 128-row blocks of M sharing each B stage, as in the
// output layer's tile passes: per FLOP a third fewer bytes land in shared memory than with one
// block) over a range of K.  When the tiles alone would leave the last wave of the grid mostly
// idle, K is split into S ranges: each unit writes its f32 partial tile to a workspace and
// gemm_split_reduce_kernel adds the S partials in a fixed order (deterministic results).
// Roles (320 threads, one CTA per SM, 225 KB of shared memory, all 512 TMEM columns):
//   warp 0, one lane: TMA producer, 3 stages of 64 KB {A block 0, A block 1, B};
//   warp 1: allocates TMEM; one lane issues tcgen05.mma (M = 128, N = 256, K = 16) into two
//     256-column accumulators and commits each stage back to the producer;
//   warps 2-9: the epilogue, one thread per row of one 128-row block (warp % 4 picks the TMEM
//     lane quarter it may read), 32 columns at a time through a per-warp shared-memory block so
//     that each store instruction writes whole 128-byte row pieces.
// Every wait is bounded (about a second): on expiry the kernel sets GRPO_DEVFLAG_TIMEOUT, the
// roles stop, in-flight copies and MMAs are drained and the tensor memory is freed.
#define GRPO_TU 7  // this file's bit in the checked build's report (grpo_debug_checks)
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "gemm.cuh"
#include "tcgen05.cuh"
#include "trace.cuh"

namespace fastrl {
namespace {

constexpr int GM = 128;  // rows of C per accumulator (MMA M, TMEM lanes); two per unit
constexpr int GN = 256;  // columns of C per unit (MMA N, TMEM columns per accumulator)
constexpr int GK = 64;   // K per stage: one 128-byte swizzle row of bf16
constexpr int kStages = 3;
constexpr uint32_t kABlockBytes = GM * GK * 2;  // 16 KB
constexpr uint32_t kBBytes = GN * GK * 2;       // 32 KB
constexpr uint32_t kBoxBytes = 64 * GK * 2;     // one MN-major box: 64 k-rows x 64 elements
constexpr uint32_t kStageBytes = 2 * kABlockBytes + kBBytes;
constexpr int kThreads = 320;
constexpr uint32_t kTmemCols = 2 * GN;
// Barriers: full and empty per stage, accumulators full and released, drain.
constexpr int kBars = 2 * kStages + 3;
constexpr uint32_t kOutWarpBytes = 32 * 32 * 4;  // per epilogue warp: 32 rows x 32 f32
constexpr size_t kSmemBytes =
    1024 + (size_t)kStages * kStageBytes + 8 * kBars + 16 + 128 + 8 * kOutWarpBytes;
static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");
constexpr uint64_t kWaitLimitNs = 1000000000ull;
constexpr int kMaxSplit = 8;

struct GemmArgs {
  int32_t M, N;
  int32_t n_mp, n_nt, nK, kb_per, S, units;
  char* C;
  int64_t ldc;
  int32_t c_bf16, accumulate, c_vec;
  float* P;  // S > 1: partial tiles [S][M][N]
  int32_t* status;
};

template <bool kAMN>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_bf16_kernel(const __grid_constant__ CUtensorMap tm_a,
                     const __grid_constant__ CUtensorMap tm_b, const GemmArgs g) {
  constexpr uint32_t kIdesc = tc::idesc_bf16(GM, GN, kAMN, true);
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw_s = smem_addr(smem_raw);
  const uint32_t base_s = (raw_s + 1023u) & ~1023u;  // swizzle atoms need 1024-byte alignment
  const uint32_t bar_s = base_s + kStages * kStageBytes;
  auto full_bar = [&](int k) { return bar_s + 8u * k; };
  auto empty_bar = [&](int k) { return bar_s + 8u * (kStages + k); };
  const uint32_t accf_bar = bar_s + 8u * (2 * kStages);
  const uint32_t acce_bar = bar_s + 8u * (2 * kStages + 1);
  const uint32_t drain_bar = bar_s + 8u * (2 * kStages + 2);
  unsigned char* tail = smem_raw + (bar_s - raw_s) + 8 * kBars;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(tail);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tail + 4);
  const uint32_t out_s = (smem_addr(tail) + 16 + 127u) & ~127u;
  // the layout (aligned stages, barriers, output staging) within the launch's shared memory
  if (!GRPO_DCHECK(out_s + 8 * kOutWarpBytes - raw_s <= dynamic_smem_bytes())) return;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int k = 0; k < kStages; ++k) {
      tc::mbar_init(full_bar(k), 1);
      tc::mbar_init(empty_bar(k), 1);
    }
    tc::mbar_init(accf_bar, 1);
    tc::mbar_init(acce_bar, 8 * 32);
    tc::mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tc::tmem_alloc(smem_addr((const void*)tmem_slot), kTmemCols);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = *tmem_slot;

  // Bounded wait; false when the phase did not complete (or another role gave up).
  auto wait_bar = [&](uint32_t bar, uint32_t parity, bool honour_abort) -> bool {
    if (tc::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1; !tc::mbar_try_wait(bar, parity); ++it) {
      if ((it & 63u) != 0) continue;
      if (honour_abort && *abort_flag) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        if (g.status) atomicOr(g.status, GRPO_DEVFLAG_TIMEOUT);
        return false;
      }
    }
    return true;
  };
  // Unit u: tile (mp, nt) of C over k-blocks [s * kb_per, min(nK, (s + 1) * kb_per)).  Units in
  // order n fastest, then m, then s: the CTAs running at once share B stages along m and A
  // stages along n in L2.
  auto unit_of = [&](int u, int& mp, int& nt, int& kb0, int& kb1) {
    nt = u % g.n_nt;
    const int r = u / g.n_nt;
    mp = r % g.n_mp;
    const int s = r / g.n_mp;
    kb0 = s * g.kb_per;
    kb1 = min(g.nK, kb0 + g.kb_per);
  };

  if (warp == 0) {
    // ---- TMA producer ----
    if (lane == 0) {
      uint32_t fills = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < g.units; u += gridDim.x) {
        int mp, nt, kb0, kb1;
        unit_of(u, mp, nt, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
          const int st = (int)(fills % kStages);
          const uint32_t ph = (fills / kStages) & 1u;
          if (!wait_bar(empty_bar(st), ph ^ 1u, true)) {
            ok = false;
            break;
          }
          const uint32_t sa = base_s + st * kStageBytes;
          const uint32_t sb = sa + 2 * kABlockBytes;
          tc::mbar_expect_tx(full_bar(st), kStageBytes);
          if (kAMN) {  // A stored [K][M]: per 128-row block, two boxes of 64 k-rows x 64 of M
#pragma unroll
            for (int b = 0; b < 2; ++b)
#pragma unroll
              for (int j = 0; j < 2; ++j)
                tc::tma_load_2d(sa + b * kABlockBytes + j * kBoxBytes, &tm_a,
                                mp * 2 * GM + b * GM + j * 64, kb * GK, full_bar(st));
          } else {  // A stored [M][K]: per block one box of 128 rows x 64 of K
            tc::tma_load_2d(sa, &tm_a, kb * GK, mp * 2 * GM, full_bar(st));
            tc::tma_load_2d(sa + kABlockBytes, &tm_a, kb * GK, mp * 2 * GM + GM, full_bar(st));
          }
#pragma unroll
          for (int j = 0; j < GN / 64; ++j)  // B stored [K][N]: four boxes of 64 k-rows x 64 of N
            tc::tma_load_2d(sb + j * kBoxBytes, &tm_b, nt * GN + j * 64, kb * GK, full_bar(st));
          ++fills;
        }
      }
      // Copies still in flight land before the CTA can exit.
      const uint32_t n = fills < (uint32_t)kStages ? fills : (uint32_t)kStages;
      for (uint32_t f = fills - n; f < fills; ++f)
        wait_bar(full_bar((int)(f % kStages)), (f / kStages) & 1u, false);
    }
  } else if (warp == 1) {
    // ---- MMA issuer ----
    if (lane == 0) {
      uint32_t fills = 0, units = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < g.units; u += gridDim.x) {
        int mp, nt, kb0, kb1;
        unit_of(u, mp, nt, kb0, kb1);
        // one accumulator pair per unit: wait until the epilogue has read the previous one
        if (!wait_bar(acce_bar, (units & 1u) ^ 1u, true)) {
          ok = false;
          break;
        }
        tc::fence_after();
        for (int kb = kb0; kb < kb1; ++kb) {
          const int st = (int)(fills % kStages);
          if (!wait_bar(full_bar(st), (fills / kStages) & 1u, true)) {
            ok = false;
            break;
          }
          tc::fence_after();
          const uint32_t sa = base_s + st * kStageBytes;
          const uint64_t bd = tc::desc_mnmajor(sa + 2 * kABlockBytes, kBoxBytes);
#pragma unroll
          for (int b = 0; b < 2; ++b) {
            const uint32_t ab = sa + b * kABlockBytes;
            const uint64_t ad = kAMN ? tc::desc_mnmajor(ab, kBoxBytes) : tc::desc_kmajor(ab);
#pragma unroll
            for (int k = 0; k < GK / 16; ++k) {
              // K = 16 per MMA: 32 bytes along a K-major row, or two 8-row atoms (2048 bytes)
              // of an MN-major box; descriptor addresses count 16-byte units.
              const uint64_t a_step = kAMN ? (uint64_t)(2048 >> 4) * k : (uint64_t)2 * k;
              tc::mma_bf16(tmem + b * GN, ad + a_step, bd + (uint64_t)(2048 >> 4) * k, kIdesc,
                           (kb != kb0 || k != 0) ? 1u : 0u);
            }
          }
          tc::commit(empty_bar(st));  // the stage is free once these MMAs have read it
          ++fills;
        }
        if (!ok) break;
        tc::commit(accf_bar);
        ++units;
      }
      // Every MMA issued has completed before the tensor memory is freed.
      tc::commit(drain_bar);
      wait_bar(drain_bar, 0, false);
    }
  } else {
    // ---- epilogue: one thread per row of one 128-row block ----
    const int q = warp & 3;            // TMEM lane quarter this warp may read
    const int half = (warp - 2) >> 2;  // which 128-row block (accumulator)
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const uint32_t blk = out_s + (uint32_t)(warp - 2) * kOutWarpBytes;
    uint32_t units = 0;
    for (int u = blockIdx.x; u < g.units; u += gridDim.x) {
      int mp, nt, kb0, kb1;
      unit_of(u, mp, nt, kb0, kb1);
      int got = 0;
      if (lane == 0) got = wait_bar(accf_bar, units & 1u, true) ? 1 : 0;
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) break;
      tc::fence_after();
      const int m0 = mp * 2 * GM + half * GM + q * 32;  // first row of this warp's 32
      const int s = kb0 / g.kb_per;
#pragma unroll 1
      for (int c = 0; c < GN; c += 32) {
        const int n0 = nt * GN + c;
        if (n0 >= g.N) break;  // warp-uniform: columns past N
        float x[32];
        tc::tmem_ld32(tmem + lane_base + half * GN + c, x);
        // this lane's row: 8 pieces of 4 values, XOR-swizzled by row (conflict-free phases)
#pragma unroll
        for (int p = 0; p < 8; ++p) {
          const uint32_t addr = blk + lane * 128u + (uint32_t)((p ^ (lane & 7)) * 16);
          asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(x[4 * p]),
                       "f"(x[4 * p + 1]), "f"(x[4 * p + 2]), "f"(x[4 * p + 3])
                       : "memory");
        }
        __syncwarp();
        // Adding to C: all eight old pieces are loaded before any is used, so that their
        // latencies overlap (loaded one by one, each behind the previous store, they held the
        // accumulators for eight round trips per piece and made an accumulating launch 25%
        // longer).  Each piece of C is read and written by this lane only.
        float4 old[8];
        const bool pre = g.S == 1 && !g.c_bf16 && g.c_vec && g.accumulate;
        if (pre) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int m = m0 + i * 4 + (lane >> 3), n = n0 + 4 * (lane & 7);
            const float4* cp = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(g.C) +
                                                               (int64_t)m * g.ldc + n);
            old[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (m < g.M && n < g.N && GRPO_DCHECK((reinterpret_cast<uintptr_t>(cp) & 15u) == 0))
              old[i] = __ldcg(cp);
          }
        }
        // 4 rows x 128 bytes per instruction: lane l takes piece l % 8 of row i * 4 + l / 8
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int rr = i * 4 + (lane >> 3), p = lane & 7;
          const uint32_t addr = blk + rr * 128u + (uint32_t)((p ^ (rr & 7)) * 16);
          float4 v;
          asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                       : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                       : "r"(addr)
                       : "memory");
          const int m = m0 + rr, n = n0 + 4 * p;
          if (m >= g.M || n >= g.N) continue;  // N is a multiple of 4: a piece is all in or out
          // the piece lies inside C (or partial s inside P), aligned for its vector store
          if (!GRPO_DCHECK(n + 4 <= g.N && (g.S > 1 ? s < g.S : m < g.M) &&
                           (g.S > 1 || !g.c_vec ||
                            ((reinterpret_cast<uintptr_t>(g.C) +
                              ((uint64_t)m * g.ldc + n) * (g.c_bf16 ? 2 : 4)) &
                             (g.c_bf16 ? 7u : 15u)) == 0)))
            continue;
          if (g.S > 1) {
            __stcg(reinterpret_cast<float4*>(g.P + ((int64_t)s * g.M + m) * g.N + n), v);
          } else if (!g.c_bf16) {
            float* cp = reinterpret_cast<float*>(g.C) + (int64_t)m * g.ldc + n;
            if (g.c_vec) {
              if (g.accumulate) {
                const float4 o = pre ? old[i] : *reinterpret_cast<const float4*>(cp);
                v.x += o.x;
                v.y += o.y;
                v.z += o.z;
                v.w += o.w;
              }
              *reinterpret_cast<float4*>(cp) = v;
            } else {
              if (g.accumulate) {
                v.x += cp[0];
                v.y += cp[1];
                v.z += cp[2];
                v.w += cp[3];
              }
              cp[0] = v.x;
              cp[1] = v.y;
              cp[2] = v.z;
              cp[3] = v.w;
            }
          } else {
            __nv_bfloat16* cp = reinterpret_cast<__nv_bfloat16*>(g.C) + (int64_t)m * g.ldc + n;
            const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y);
            const __nv_bfloat162 hi = __floats2bfloat162_rn(v.z, v.w);
            if (g.c_vec) {
              *reinterpret_cast<uint2*>(cp) = make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                                                         *reinterpret_cast<const uint32_t*>(&hi));
            } else {
              cp[0] = lo.x;
              cp[1] = lo.y;
              cp[2] = hi.x;
              cp[3] = hi.y;
            }
          }
        }
        __syncwarp();
      }
      tc::fence_before();
      tc::mbar_arrive(acce_bar);
      ++units;
    }
  }

  __syncwarp();  // lanes that had no role wait for their warp's working lane
  tc::fence_before();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// C[m, n] = P[0][m][n] + ... + P[S-1][m][n] (+ the old C), in that order; 4 columns per thread.
__global__ void __launch_bounds__(256) gemm_split_reduce_kernel(const float4* __restrict__ P,
                                                                int32_t S, int32_t M, int32_t N,
                                                                char* C, int64_t ldc,
                                                                int32_t c_bf16, int32_t accumulate,
                                                                int32_t c_vec) {
  const int64_t n4 = N / 4;
  const int64_t total = (int64_t)M * n4;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    float4 v = __ldcs(P + i);
    for (int s = 1; s < S; ++s) {
      const float4 o = __ldcs(P + (int64_t)s * total + i);
      v.x += o.x;
      v.y += o.y;
      v.z += o.z;
      v.w += o.w;
    }
    const int64_t m = i / n4, n = (i % n4) * 4;
    if (!c_bf16) {
      float* cp = reinterpret_cast<float*>(C) + m * ldc + n;
      if (accumulate) {
        v.x += cp[0];
        v.y += cp[1];
        v.z += cp[2];
        v.w += cp[3];
      }
      if (c_vec) {
        *reinterpret_cast<float4*>(cp) = v;
      } else {
        cp[0] = v.x;
        cp[1] = v.y;
        cp[2] = v.z;
        cp[3] = v.w;
      }
    } else {
      __nv_bfloat16* cp = reinterpret_cast<__nv_bfloat16*>(C) + m * ldc + n;
      const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y);
      const __nv_bfloat162 hi = __floats2bfloat162_rn(v.z, v.w);
      if (c_vec) {
        *reinterpret_cast<uint2*>(cp) = make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                                                   *reinterpret_cast<const uint32_t*>(&hi));
      } else {
        cp[0] = lo.x;
        cp[1] = lo.y;
        cp[2] = hi.x;
        cp[3] = hi.y;
      }
    }
  }
}

}  // namespace

// K split: the S that minimises the CTAs' busiest share of (k-blocks + a per-unit overhead)
// plus the partials' extra HBM traffic, counted in k-block times (one k-block of a unit is
// 2 * 256 * 256 * 64 FLOPs, about 0.73 us per SM at the measured rate; HBM moves about
// 6 GB/s per microsecond).  A larger S must gain more than 1%.
GemmPlan gemm_plan(int64_t M, int64_t N, int64_t K, int n_sm) {
  GemmPlan p;
  const int64_t n_mp = (M + 2 * GM - 1) / (2 * GM), n_nt = (N + GN - 1) / GN;
  const int64_t nK = std::max<int64_t>(1, (K + GK - 1) / GK);
  const int64_t tiles = n_mp * n_nt;
  const int64_t sms = std::max(n_sm, 1);
  const double kb_us = 0.73, unit_overhead_kb = 6.0, hbm_bytes_per_us = 6.0e6;
  double best = -1.0;
  p.S = 1;
  p.kb_per = (int)nK;
  for (int S = 1; S <= kMaxSplit; ++S) {
    const int64_t kb_per = (nK + S - 1) / S;
    if (S > 1 && kb_per < 16) break;
    const int64_t Sr = (nK + kb_per - 1) / kb_per;  // every range holds at least one k-block
    if (Sr != S) continue;
    const int64_t units = Sr * tiles;
    const int64_t waves = (units + sms - 1) / sms;
    double cost = (double)waves * ((double)kb_per + unit_overhead_kb);
    if (Sr > 1) cost += (double)(Sr + 1) * M * N * 4 / hbm_bytes_per_us / kb_us;
    if (best < 0.0 || cost < best * 0.99) {
      best = cost;
      p.S = (int)Sr;
      p.kb_per = (int)kb_per;
    }
  }
  p.units = p.S * tiles;
  p.grid = (int)std::min<int64_t>(p.units, sms);
  p.partial_bytes = p.S > 1 ? (size_t)p.S * M * N * sizeof(float) : 0;
  return p;
}

grpo_status gemm_bf16(const char* who, bool a_mn, const void* A, int64_t lda, const void* B,
                      int64_t ldb, int64_t M, int64_t N, int64_t K, void* C, int64_t ldc,
                      int32_t c_dtype, bool accumulate, float* partial, size_t partial_bytes,
                      int32_t* status, cudaStream_t s) {
  if (M <= 0 || N <= 0 || K <= 0 || M >= ((int64_t)1 << 31) || N >= ((int64_t)1 << 31) ||
      K >= ((int64_t)1 << 31) || N % 4 != 0 || lda % 8 != 0 || ldb % 8 != 0 || ldc < N ||
      ((uintptr_t)A | (uintptr_t)B) % 16 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: GEMM %lld x %lld x %lld with lda %lld ldb %lld ldc %lld",
                who, (long long)M, (long long)N, (long long)K, (long long)lda, (long long)ldb,
                (long long)ldc);
  if (accumulate && c_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: accumulation needs an f32 output", who);
  const size_t esz = c_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  if (C == nullptr || (uintptr_t)C % esz != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: output not aligned to its element size", who);
  const int n_sm = tc::sm_count();
  if (n_sm <= 0) return fail(GRPO_ERR_CUDA, "%s: no CUDA device", who);
  GemmPlan p = gemm_plan(M, N, K, n_sm);
  if (p.S > 1 && (partial == nullptr || partial_bytes < p.partial_bytes ||
                  (uintptr_t)partial % 16 != 0)) {
    p.S = 1;  // no room for the partials: run unsplit
    p.kb_per = (int)((K + GK - 1) / GK);
    p.units = (int)(((M + 2 * GM - 1) / (2 * GM)) * ((N + GN - 1) / GN));
    p.grid = std::min(p.units, n_sm);
  }
  CUtensorMap ma, mb;
  const bool ok_a = a_mn ? tc::make_map_bf16(&ma, A, K, M, lda, 64)    // [K][M], boxes 64 x 64
                         : tc::make_map_bf16(&ma, A, M, K, lda, GM);   // [M][K], boxes 128 x 64
  if (!ok_a || !tc::make_map_bf16(&mb, B, K, N, ldb, 64))
    return fail(GRPO_ERR_CUDA, "%s: cuTensorMapEncodeTiled failed", who);
  GemmArgs g = {};
  g.M = (int32_t)M;
  g.N = (int32_t)N;
  g.n_mp = (int32_t)((M + 2 * GM - 1) / (2 * GM));
  g.n_nt = (int32_t)((N + GN - 1) / GN);
  g.nK = (int32_t)((K + GK - 1) / GK);
  g.kb_per = p.kb_per;
  g.S = p.S;
  g.units = p.units;
  g.C = static_cast<char*>(C);
  g.ldc = ldc;
  g.c_bf16 = c_dtype == GRPO_DTYPE_BF16 ? 1 : 0;
  g.accumulate = accumulate ? 1 : 0;
  g.c_vec = ((uintptr_t)C % (4 * esz) == 0 && (ldc * esz) % (4 * esz) == 0) ? 1 : 0;
  g.P = p.S > 1 ? partial : nullptr;
  g.status = status;

  // The shared-memory limit is a per-device function attribute: set it once on each device.
  static std::mutex mu;
  static uint64_t done = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: cudaGetDevice: %s", who, cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return fail(GRPO_ERR_UNSUPPORTED, "%s: device %d beyond 64", who, dev);
  {
    std::lock_guard<std::mutex> lk(mu);
    if (!((done >> dev) & 1u)) {
      e = cudaFuncSetAttribute(gemm_bf16_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)kSmemBytes);
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(gemm_bf16_kernel<true>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
      if (e != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "%s: cudaFuncSetAttribute: %s", who, cudaGetErrorString(e));
      done |= uint64_t(1) << dev;
    }
  }
  if (a_mn)
    gemm_bf16_kernel<true><<<p.grid, kThreads, kSmemBytes, s>>>(ma, mb, g);
  else
    gemm_bf16_kernel<false><<<p.grid, kThreads, kSmemBytes, s>>>(ma, mb, g);
  count_launches(1);
  grpo_status st = check_launch(who);
  if (st != GRPO_OK || p.S == 1) return st;
  const int64_t work = M * (N / 4);
  const int blocks = (int)std::min<int64_t>((work + 255) / 256, (int64_t)n_sm * 8);
  gemm_split_reduce_kernel<<<blocks, 256, 0, s>>>(reinterpret_cast<const float4*>(partial), p.S,
                                                  (int32_t)M, (int32_t)N, static_cast<char*>(C),
                                                  ldc, g.c_bf16, g.accumulate, g.c_vec);
  count_launches(1);
  return check_launch(who);
}

}  // namespace fastrl

using namespace fastrl;

extern "C" grpo_status grpo_lmhead_grad(const void* dlogits, int64_t dlogits_stride, int64_t n_rows,
                                        int32_t V, const void* hidden, int64_t hidden_stride,
                                        const void* weight, int32_t D, void* dhidden,
                                        int32_t dhidden_dtype, float* dweight,
                                        int32_t accumulate_dweight, int32_t* status, void* ws,
                                        size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_lmhead_grad");
  clear_error();
  const char* who = "grpo_lmhead_grad";
  if (n_rows < 0 || n_rows >= ((int64_t)1 << 31) || V < 1 || D < 8 || D % 8 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: need n_rows in [0, 2^31), V >= 1, D a positive "
                "multiple of 8 (n_rows=%lld V=%d D=%d)", who, (long long)n_rows, V, D);
  if (dlogits_stride < V || dlogits_stride % 8 != 0 || hidden_stride < D || hidden_stride % 8 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: strides must be multiples of 8, dlogits_stride >= V and "
                "hidden_stride >= D (%lld, %lld)", who, (long long)dlogits_stride,
                (long long)hidden_stride);
  if (dhidden_dtype != GRPO_DTYPE_BF16 && dhidden_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: dhidden_dtype must be BF16 or F32", who);
  int n_sm = tc::sm_count();
  if (n_sm <= 0) n_sm = 152;  // a size query on a machine without a device
  size_t need = 0;
  if (n_rows > 0) {
    if (dhidden) need = std::max(need, gemm_plan(n_rows, D, V, n_sm).partial_bytes);
    if (dweight) need = std::max(need, gemm_plan(V, D, n_rows, n_sm).partial_bytes);
  }
  need = align_up(need, 256);
  bool query = false;
  grpo_status st = workspace_check(ws, ws_bytes, need, who, &query);
  if (st != GRPO_OK || query) return st;
  cudaStream_t s = as_stream(stream);
  if (n_rows == 0) {  // no rows: dhidden is empty, dweight is 0 (or unchanged when accumulated)
    if (dweight && !accumulate_dweight) {
      const cudaError_t e = cudaMemsetAsync(dweight, 0, (size_t)V * D * sizeof(float), s);
      if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
    }
    return GRPO_OK;
  }
  if (!dlogits || (dhidden && !weight) || (dweight && !hidden))
    return fail(GRPO_ERR_INVALID_ARG, "%s: a required pointer is NULL", who);
  if (((uintptr_t)dlogits | (uintptr_t)hidden | (uintptr_t)weight) % 16 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: dlogits, hidden and weight must be 16-byte aligned", who);
  float* part = static_cast<float*>(ws);
  if (dhidden &&
      (st = gemm_bf16(who, false, dlogits, dlogits_stride, weight, D, n_rows, D, V, dhidden, D,
                      dhidden_dtype, false, part, need, status, s)) != GRPO_OK)
    return st;
  if (dweight &&
      (st = gemm_bf16(who, true, dlogits, dlogits_stride, hidden, hidden_stride, V, D, n_rows,
                      dweight, D, GRPO_DTYPE_F32, accumulate_dweight != 0, part, need, status,
                      s)) != GRPO_OK)
    return st;
  return GRPO_OK;
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_gemm)
}  // namespace fastrl
