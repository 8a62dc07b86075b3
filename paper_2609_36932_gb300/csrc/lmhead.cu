// The policy's output layer fused with the GRPO token loss, on the tensor cores.
//
// Sec. 3.2 runs every kept trajectory through the policy, whose last layer maps each token's
// hidden state h_t (D values) to logits over the vocabulary; Eqs. 1-3 turn those into the loss.
// With the output layer's weight rows W_v:
//   z[t, v] = sum_d h[t, d] * W[v, d]
//   loss, logp: Eqs. 1-3 on z, as grpo_loss_fwd_bwd computes them
//   dh = dlogits * W,   dW = dlogits^T * h        (the chain rule through z = h W^T)
// The [rows, V] logits never exist for all rows at once.  They are produced 128 x 256 at a time
// into tensor memory by tcgen05.mma (bf16 operands staged in shared memory by TMA, f32
// accumulators).
// The token loss runs chunk by chunk (rows of logits held at a time):
//   Pass 1 (lmhead_tile_kernel<false>): per row and vocabulary tile, the maximum and the sum of
//     exp(z - max) (z_y excluded from the sum and kept separately); the chunk's f32 logits are
//     stored as they leave tensor memory.
//   lmhead_rows_kernel: the per-tile sums combined in a fixed order -> lse, logp, the loss term
//     and the gradient scalars of each row (the same formulas as the fused loss kernel).
//   lmhead_dlogits_kernel: dlogits = coef * ([v == y] - softmax(z)_v) in bf16 from the stored
//     logits, a streaming pass (6 bytes per entry instead of a second 2 D FLOPs per entry).
//   Two products per chunk on the same tensor-core machinery (gemm.cu): dh = dlogits * W and
//     dW (+)= dlogits^T * h.
// GSPO's loss couples every row of a sequence, and a sequence may cross a chunk boundary, so its
// entry runs pass 1 over every row first, keeping the first chunk's f32 logits; that chunk's
// dlogits come from them, and each later chunk's from pass 2 (lmhead_tile_kernel<true>), which
// recomputes the tiles and writes dlogits from tensor memory.  grpo_lmhead_tune can select the
// recomputation for every chunk of both losses (less workspace: no chunk of f32 logits).
//
// Kernel roles (320 threads, one CTA per SM: 225 KB of shared memory, all 512 TMEM columns).  A
// tile is a pair of 128-row blocks of h against 256 vocabulary entries, so each weight stage
// feeds two row blocks: per FLOP a third fewer bytes land in shared memory than with one row
// block per tile, which on GB300 made the kernel 5.5% faster (shared-memory traffic, not the
// tensor core, was its limit), at the price of a single pair of accumulators.
//   warp 0, one lane: TMA producer, 3 stages of {A0, A1: 128 rows x 64 of h each, B: 256 rows x
//     64 of W}, 128-byte swizzled;
//   warp 1: allocates TMEM; one lane issues the MMAs (M = 128, N = 256, K = 16) into two
//     256-column accumulators, one per row block of the pair;
//   warps 2-9: the epilogue, one thread per row of one row block (warps 2-5 the first, 6-9 the
//     second), reading its row from TMEM 32 columns at a time (a warp may read only its quarter of
//     the 128 lanes: warp % 4).  The next tile's MMAs wait for it to release the accumulators.
// Work: CTA c owns pair lane i = c % R and vocabulary lane j = c / R; for each group of R row-block
// pairs it takes pair g*R + i and the vocabulary tiles j, j + J, j + 2J, ...  At any time the grid
// works on 2R consecutive row blocks and J consecutive vocabulary tiles, which the L2 serves to
// all of it; the weight streams from DRAM about once per group (R = 4..8 pairs, chosen per
// launch for the fewest idle CTAs).  Pass 1 stages each warp's 32 x 32 block of f32 logits in
// shared memory and writes it as 128-byte row pieces; pass 2 its 32 x 32 block of dlogits as
// 64-byte row pieces (1.3% faster than 16-byte pieces straight from the registers); both with
// streaming stores so that they do not displace the operand tiles in L2.  An L2 prefetch of
// upcoming tiles (grpo_lmhead_tune) is off by default: on GB300 it made pass 1 about 16% slower.
//
// Every wait is bounded (about a second): a wait that runs out sets GRPO_DEVFLAG_TIMEOUT and an
// abort flag; the roles then stop, the producer waits for its copies in flight and the MMA lane
// for its MMAs, and warp 1 frees the tensor memory before the CTA exits.
#define GRPO_TU 6  // this file's bit in the checked build's report (grpo_debug_checks)
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "gemm.cuh"
#include "tcgen05.cuh"
#include "trace.cuh"
#include "rowops.cuh"

namespace fastrl {
namespace {

constexpr int BM = 128;  // rows of h per row block (MMA M; TMEM lanes); two blocks per tile
constexpr int BN = 256;  // vocabulary entries per tile (MMA N; TMEM columns per accumulator)
constexpr int BK = 64;   // D per stage: one 128-byte swizzle row of bf16
constexpr int kStages = 3;
constexpr uint32_t kABytes = BM * BK * 2;
constexpr uint32_t kBBytes = BN * BK * 2;
constexpr uint32_t kStageBytes = 2 * kABytes + kBBytes;  // two row blocks share B
constexpr int kThreads = 320;
constexpr uint32_t kTmemCols = 2 * BN;  // one accumulator per row block of the pair
constexpr int kRowLanes = 8;       // R: row-block pairs in flight across the grid
constexpr int kMaxJ = 160;         // vocabulary lanes at most
// Barriers: full and empty per stage, accumulator-pair full and released (two slots each, the
// first in use), drain.
constexpr int kBars = 2 * kStages + 5;
// Output staging per epilogue warp: 32 rows x 128 bytes (32 f32 logits in pass 1, 32 bf16 dlogits
// in pass 2, which uses the first half).
constexpr uint32_t kStageWarpBytes = 32 * 128;
constexpr uint32_t kStageOutBytes = 8 * kStageWarpBytes;
constexpr size_t kSmemBytes = 1024 + (size_t)kStages * kStageBytes + 8 * kBars + 16 + 128 +
                              kStageOutBytes;
static_assert(kSmemBytes <= 227 * 1024, "the tile kernel's shared memory exceeds a CTA's limit");
constexpr uint64_t kWaitLimitNs = 1000000000ull;
constexpr int64_t kDefaultChunkBytes = 4ll << 30;  // dlogits chunk buffer

// Instruction descriptor of tcgen05.mma.kind::f16 for the tile passes: f32 accumulator, bf16 A
// (h) and B (W), both K-major (D contiguous), N = BN, M = BM.
constexpr uint32_t kIdesc = tc::idesc_bf16(BM, BN, false, false);

using tc::mbar_arrive;
using tc::mbar_expect_tx;
using tc::mbar_init;
using tc::mbar_try_wait;
using tc::tma_load_2d;
using tc::tma_prefetch_2d;
using tc::tmem_ld32;
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) { return tc::desc_kmajor(saddr); }
__device__ __forceinline__ void tc_fence_before() { tc::fence_before(); }
__device__ __forceinline__ void tc_fence_after() { tc::fence_after(); }
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                       uint32_t accumulate) {
  tc::mma_bf16(d_tmem, adesc, bdesc, kIdesc, accumulate);
}
__device__ __forceinline__ void tc_commit(uint32_t bar) { tc::commit(bar); }

struct TileArgs {
  int32_t rows;   // rows of this launch (a chunk in pass 2); the tensor map's row = row0 + local
  int32_t row0;
  int32_t V, nK, n_vt, n_rb, R, J;
  int32_t prefetch;  // k-blocks between a tile's L2 prefetch and its load (0: none)
  // n_rb counts row blocks; tiles take them in pairs (2p, 2p + 1)
  const int32_t* y;  // [rows]
  // pass 1
  float2* part;  // [rows][n_vt]: (max, sum of exp(z - max) without z_y) of vocabulary tile vt
  float* zy;     // [rows]: z_y, written by the CTA whose tile holds y
  float* z;      // nullable [z_rows][ldz]: the f32 logits of rows < z_rows, for the dlogits pass
  int64_t ldz;
  int32_t z_rows;  // a multiple of 32 (or rows)
  // pass 2
  const float4* rowsc;  // [rows]: {neg_scale, dy, shift, 0} from lmhead_rows_kernel
  __nv_bfloat16* dl;    // [rows][ldd]
  int64_t ldd;
  int32_t* status;
};

template <bool kBwd>
__global__ void __launch_bounds__(kThreads, 1)
    lmhead_tile_kernel(const __grid_constant__ CUtensorMap tm_h,
                       const __grid_constant__ CUtensorMap tm_w, const TileArgs a) {
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw_s = smem_addr(smem_raw);
  const uint32_t base_s = (raw_s + 1023u) & ~1023u;  // swizzle atoms need 1024-byte alignment
  const uint32_t bar_s = base_s + kStages * kStageBytes;
  auto full_bar = [&](int k) { return bar_s + 8u * k; };
  auto empty_bar = [&](int k) { return bar_s + 8u * (kStages + k); };
  auto accf_bar = [&](int k) { return bar_s + 8u * (2 * kStages + k); };
  auto acce_bar = [&](int k) { return bar_s + 8u * (2 * kStages + 2 + k); };
  const uint32_t drain_bar = bar_s + 8u * (2 * kStages + 4);
  unsigned char* tail = smem_raw + (bar_s - raw_s) + 8 * kBars;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(tail);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tail + 4);
  // output staging: kStageWarpBytes per epilogue warp, 128-byte aligned
  const uint32_t stage_out_s = (smem_addr(tail) + 16 + 127u) & ~127u;
  // the layout (aligned stages, barriers, output staging) within the launch's shared memory
  if (!GRPO_DCHECK(stage_out_s + kStageOutBytes - raw_s <= dynamic_smem_bytes())) return;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int k = 0; k < kStages; ++k) {
      mbar_init(full_bar(k), 1);
      mbar_init(empty_bar(k), 1);
    }
    for (int k = 0; k < 2; ++k) {
      mbar_init(accf_bar(k), 1);
      mbar_init(acce_bar(k), 8 * 32);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr((const void*)tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Bounded wait; false when the phase did not complete (or another role gave up).
  auto wait_bar = [&](uint32_t bar, uint32_t parity, bool honour_abort) -> bool {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1; !mbar_try_wait(bar, parity); ++it) {
      if ((it & 63u) != 0) continue;
      if (honour_abort && *abort_flag) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        if (a.status) atomicOr(a.status, GRPO_DEVFLAG_TIMEOUT);
        return false;
      }
    }
    return true;
  };

  const int R = a.R, J = a.J;
  const int li = (int)blockIdx.x % R, lj = (int)blockIdx.x / R;

  if (warp == 0) {
    // ---- TMA producer ----
    if (lane == 0) {
      uint32_t fills = 0;
      bool ok = true;
      // A second walk over the same (row block, vocabulary tile, k-block) sequence, a.prefetch
      // fills ahead of the loads, asks L2 for those tiles early.
      const int n_rp = (a.n_rb + 1) / 2;
      int prb = li, pvt = lj, pkb = 0;
      auto advance = [&]() {
        if (++pkb == a.nK) {
          pkb = 0;
          pvt += J;
          if (pvt >= a.n_vt) {
            pvt = lj;
            prb += R;
          }
        }
      };
      for (int k = 0; k < a.prefetch && prb < n_rp; ++k) advance();
      for (int rp = li; ok && rp < n_rp; rp += R) {
        const int rb = 2 * rp;
        for (int vt = lj; ok && vt < a.n_vt; vt += J) {
          for (int kb = 0; kb < a.nK; ++kb) {
            const int st = (int)(fills % kStages);
            const uint32_t ph = (fills / kStages) & 1u;
            if (!wait_bar(empty_bar(st), ph ^ 1u, true)) {
              ok = false;
              break;
            }
            const uint32_t sa = base_s + st * kStageBytes;
            mbar_expect_tx(full_bar(st), kStageBytes);
            tma_load_2d(sa, &tm_h, kb * BK, a.row0 + rb * BM, full_bar(st));
            tma_load_2d(sa + kABytes, &tm_h, kb * BK, a.row0 + (rb + 1) * BM, full_bar(st));
            tma_load_2d(sa + 2 * kABytes, &tm_w, kb * BK, vt * BN, full_bar(st));
            ++fills;
            if (a.prefetch > 0 && prb < n_rp) {
              tma_prefetch_2d(&tm_h, pkb * BK, a.row0 + 2 * prb * BM);
              tma_prefetch_2d(&tm_h, pkb * BK, a.row0 + (2 * prb + 1) * BM);
              tma_prefetch_2d(&tm_w, pkb * BK, pvt * BN);
              advance();
            }
          }
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
      uint32_t fills = 0, tiles = 0;
      bool ok = true;
      const int n_rp = (a.n_rb + 1) / 2;
      for (int rp = li; ok && rp < n_rp; rp += R) {
        for (int vt = lj; ok && vt < a.n_vt; vt += J) {
          // one accumulator pair (256 columns per row block) per tile: wait until the epilogue
          // has read the previous tile's
          if (!wait_bar(acce_bar(0), (tiles & 1u) ^ 1u, true)) {
            ok = false;
            break;
          }
          tc_fence_after();
          for (int kb = 0; kb < a.nK; ++kb) {
            const int st = (int)(fills % kStages);
            if (!wait_bar(full_bar(st), (fills / kStages) & 1u, true)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = base_s + st * kStageBytes;
            const uint64_t ad0 = smem_desc(sa), ad1 = smem_desc(sa + kABytes);
            const uint64_t bd = smem_desc(sa + 2 * kABytes);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)  // K = 16 per MMA: 32 bytes along the swizzled row
              tc_mma(tmem, ad0 + 2 * k, bd + 2 * k, (kb | k) != 0 ? 1u : 0u);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)
              tc_mma(tmem + BN, ad1 + 2 * k, bd + 2 * k, (kb | k) != 0 ? 1u : 0u);
            tc_commit(empty_bar(st));  // the stage is free once these MMAs have read it
            ++fills;
          }
          if (!ok) break;
          tc_commit(accf_bar(0));
          ++tiles;
        }
      }
      // Every MMA issued has completed before the tensor memory is freed.
      tc_commit(drain_bar);
      wait_bar(drain_bar, 0, false);
    }
  } else {
    // ---- epilogue: one thread per tile row ----
    const int q = warp & 3;            // TMEM lane quarter this warp may read
    const int half = (warp - 2) >> 2;  // which row block (accumulator) of the pair
    const int r_in = q * 32 + lane;    // row within the row block
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    uint32_t tiles = 0;
    bool ok = true;
    const int n_rp = (a.n_rb + 1) / 2;
    for (int rp = li; ok && rp < n_rp; rp += R) {
      const int rb = 2 * rp + half;
      const int row = rb * BM + r_in;
      const bool rv = row < a.rows;
      const int yv = rv ? a.y[row] : -1;
      float4 sc = make_float4(0.f, 0.f, 0.f, 0.f);
      if (kBwd && rv) sc = a.rowsc[row];
      const float neg_scale = sc.x, dy = sc.y, shB = sc.z;
      const uint32_t blk = stage_out_s + (uint32_t)(warp - 2) * kStageWarpBytes;
      for (int vt = lj; vt < a.n_vt; vt += J) {
        // pass 1: this tile's maximum and sum of exp(z - m) without z_y
        float m = -INFINITY, s = 0.f;
        int got = 0;
        if (lane == 0) got = wait_bar(accf_bar(0), tiles & 1u, true) ? 1 : 0;
        got = __shfl_sync(0xffffffffu, got, 0);
        if (!got) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr = tmem + lane_base + half * BN;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int v0 = vt * BN + c;
          if (v0 >= a.V) break;  // warp-uniform: columns past the vocabulary
          float x[32];
          tmem_ld32(taddr + c, x);
          const int nvalid = a.V - v0;  // >= 1
          const int jy = yv - v0;       // y's column in this chunk, if in [0, 32)
          if (!kBwd) {
            if (a.z != nullptr && rb * BM + q * 32 < a.z_rows) {  // warp-uniform
              // The row's 32 logits through shared memory (16-byte pieces XOR-swizzled by row,
              // conflict-free), then each store instruction covers 4 rows x 128 contiguous bytes.
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const uint32_t addr = blk + lane * 128u + (uint32_t)((k ^ (lane & 7)) * 16);
                asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                             "f"(x[4 * k]), "f"(x[4 * k + 1]), "f"(x[4 * k + 2]),
                             "f"(x[4 * k + 3])
                             : "memory");
              }
              __syncwarp();
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const int rr = i * 4 + (lane >> 3);  // row within the warp's 32
                const int kc = lane & 7;             // 16-byte piece of that row
                const uint32_t addr = blk + rr * 128u + (uint32_t)((kc ^ (rr & 7)) * 16);
                float4 v;
                asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                             : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                             : "r"(addr)
                             : "memory");
                const int grow = rb * BM + q * 32 + rr;
                // streaming: the logits must not push the operands out of L2
                if (grow < a.rows && grow < a.z_rows && GRPO_DCHECK(v0 + 32 <= a.ldz))
                  __stcs(reinterpret_cast<float4*>(a.z + (int64_t)grow * a.ldz + v0) + kc, v);
              }
              __syncwarp();
            }
            float cm = -INFINITY;
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              if (k >= nvalid) x[k] = -INFINITY;
              cm = fmaxf(cm, x[k]);
            }
            if (cm > m) {
              s *= ex2((m - cm) * kLog2e);
              m = cm;
            }
            const float mb = m * kLog2e;
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int k = 0; k < 32; k += 2) {
              const float e0 = (k == jy) ? 0.f : ex2(fmaf(x[k], kLog2e, -mb));
              const float e1 = (k + 1 == jy) ? 0.f : ex2(fmaf(x[k + 1], kLog2e, -mb));
              s0 += e0;
              s1 += e1;
            }
            s += s0 + s1;
            if (rv && (unsigned)jy < 32u) {
              float zyv = 0.f;
#pragma unroll
              for (int k = 0; k < 32; ++k)
                if (k == jy) zyv = x[k];
              a.zy[row] = zyv;
            }
          } else {
            uint32_t pk[16];
#pragma unroll
            for (int k = 0; k < 32; k += 2) {
              float d0 = neg_scale * ex2(fmaf(x[k], kLog2e, shB));
              float d1 = neg_scale * ex2(fmaf(x[k + 1], kLog2e, shB));
              if (k == jy) d0 = dy;
              if (k + 1 == jy) d1 = dy;
              if (k >= nvalid) d0 = 0.f;
              if (k + 1 >= nvalid) d1 = 0.f;
              pk[k / 2] = pack_bf16x2(make_float2(d0, d1));
            }
            // Through shared memory: each lane writes its row's 64 bytes (16-byte pieces XOR-
            // swizzled by row, conflict-free), then each store instruction covers 8 rows x 64
            // contiguous bytes instead of 32 rows x 16 bytes.
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint32_t addr = blk + lane * 64u + (uint32_t)((k ^ ((lane >> 1) & 3)) * 16);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                           "r"(pk[4 * k]), "r"(pk[4 * k + 1]), "r"(pk[4 * k + 2]),
                           "r"(pk[4 * k + 3])
                           : "memory");
            }
            __syncwarp();
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int rr = i * 8 + (lane >> 2);  // row within the warp's 32
              const int kc = lane & 3;             // 16-byte piece of that row
              const uint32_t addr = blk + rr * 64u + (uint32_t)((kc ^ ((rr >> 1) & 3)) * 16);
              uint4 v;
              asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                           : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                           : "r"(addr)
                           : "memory");
              const int grow = rb * BM + q * 32 + rr;
              // streaming: dlogits must not push the operand tiles out of L2
              if (grow < a.rows && GRPO_DCHECK(v0 + 32 <= a.ldd))
                __stcs(reinterpret_cast<uint4*>(a.dl + (int64_t)grow * a.ldd + v0) + kc, v);
            }
            __syncwarp();
          }
        }
        tc_fence_before();
        mbar_arrive(acce_bar(0));
        ++tiles;
        if (!kBwd && rv) a.part[(int64_t)row * a.n_vt + vt] = make_float2(m, s);
      }
    }
  }

  __syncwarp();  // lanes that had no role wait for their warp's working lane
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

struct RowArgs {
  int32_t rows, n_vt, V;
  const float2* part;  // [rows][n_vt]
  const float* zy;
  const int32_t* y;
  const float *old_logp, *ref_logp, *adv;
  const int32_t* row_rollout;
  const int64_t* seq_off;
  float beta, lo_up, hi_dn, lo_rn, hi_rn;
  int32_t agg_mode;
  double inv_denom;
  float inv_denom_f, inv_nseq_f;
  float* logp_out;
  double* row_loss;
  float4* rowsc;
  int32_t* status;
  // 0: the token loss (row_loss, rowsc); 1: logp_out alone; 2: logp_out and the softmax
  // statistics {M, S, S without y, 0} in stats, for GSPO's sequence kernel
  int32_t mode;
  float4* stats;
};

constexpr int kRowWarps = 8;

// One warp per row: combine the row's per-tile partial sums, then apply Eqs. 1-3 in lane 0 (the
// same arithmetic as the fused loss kernel's row scalars).  Lane l takes tiles l, l + 32, ...,
// and the lanes' values meet in a fixed xor tree, so the result depends only on the row's
// logits: not on how pass 1's grid visited the tiles, nor on how the rows were chunked.
__global__ void __launch_bounds__(kRowWarps * 32) lmhead_rows_kernel(const RowArgs a) {
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
  if (t >= a.rows) return;
  const int yv = a.y[t];
  if (yv < 0 || yv >= a.V) {
    if (lane != 0) return;
    if (a.logp_out) a.logp_out[t] = __int_as_float(0x7fc00000);
    if (a.mode == 0) {
      a.row_loss[t] = 0.0;
      a.rowsc[t] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (a.status) atomicOr(a.status, GRPO_DEVFLAG_BAD_TOKEN);
    return;
  }
  const float2* p = a.part + (int64_t)t * a.n_vt;
  float M = -INFINITY;
  for (int j = lane; j < a.n_vt; j += 32) M = fmaxf(M, p[j].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float S_excl = 0.f;
  for (int j = lane; j < a.n_vt; j += 32) {
    const float2 v = p[j];
    if (v.x != -INFINITY) S_excl += v.y * expf(v.x - M);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) S_excl += __shfl_xor_sync(0xffffffffu, S_excl, o);
  if (lane != 0) return;
  const float zy = a.zy[t];
  const float S = S_excl + expf(zy - M);
  const float logp = (zy - M) - logf(S);
  if (a.mode != 0) {
    a.logp_out[t] = logp;
    if (a.mode == 2) a.stats[t] = make_float4(M, S, S_excl, 0.f);
    if (a.status && !isfinite(logp)) atomicOr(a.status, GRPO_DEVFLAG_NONFINITE);
    return;
  }
  const float A = a.adv[a.row_rollout[t]];
  const float rho = expf(logp - a.old_logp[t]);
  const float clipped = rho < a.lo_up ? a.lo_rn : (rho > a.hi_dn ? a.hi_rn : rho);
  const float surr = fminf(rho * A, clipped * A);
  const float x = a.ref_logp[t] - logp;
  const float em1 = expm1f(x);
  const float kl = em1 - x;
  const float ell = -(surr - a.beta * kl);
  float w;
  if (a.agg_mode == 0) {
    w = a.inv_denom_f;
  } else {
    const int32_t r = a.row_rollout[t];
    w = a.inv_nseq_f / (float)(a.seq_off[r + 1] - a.seq_off[r]);
  }
  const bool c = (A >= 0.f) ? (rho <= a.hi_dn) : (rho >= a.lo_up);
  const float g = -((c ? rho * A : 0.f) + a.beta * em1);
  const float coef = w * g;
  float neg_scale = -coef / S;
  const float dy = coef * (S_excl / S);
  float shB = -M * kLog2e;
  if (fabsf(neg_scale) >= 0x1p-100f) {
    shB += kShiftB;
    neg_scale *= 0x1p-16f;  // 2^-kShiftB
  }
  a.rowsc[t] = make_float4(neg_scale, dy, shB, 0.f);
  if (a.logp_out) a.logp_out[t] = logp;
  a.row_loss[t] = (a.agg_mode == 0 ? a.inv_denom : (double)w) * (double)ell;
  if (a.status && !isfinite(logp)) atomicOr(a.status, GRPO_DEVFLAG_NONFINITE);
}

struct SeqArgs {
  const float* logp;  // rows in order (after any gather)
  const float* old_logp;
  const float* ref_logp;
  const float* adv;
  const int32_t* seq_rollout;
  const int64_t* seq_row_off;
  int32_t n_seq_rows;
  int64_t n_rows;
  double lo, hi;  // 1 - eps_low, 1 + eps_high
  float beta;
  double inv_nseq;
  const float4* stats;
  float4* rowsc;
  double* seq_loss;
  float* seq_ratio;
};

constexpr int kSeqWarps = 8;

// GSPO's sequence-level ratio (Sec. 1, Sec. 4: FastRL on GSPO), one warp per sequence k with rows
// [r0, r1):  log s_k = mean_t(logp_t - old_t), clipped per sequence; the sequence's loss term and
// each row's gradient scalars for pass 2 (coef_t = w_t g_t turned into {neg_scale, dy, shift} as
// in lmhead_rows_kernel).  fp64 lane sums combined by a fixed xor tree: the result depends only on
// the sequence's rows.  A sequence with a non-finite logp (an invalid token) or no rows has no
// ratio: loss term 0, ratio NaN, zero gradient.
__global__ void __launch_bounds__(kSeqWarps * 32) lmhead_gspo_seq_kernel(const SeqArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t k = (int64_t)blockIdx.x * kSeqWarps + (threadIdx.x >> 5);
  if (k >= a.n_seq_rows) return;
  int64_t r0 = a.seq_row_off[k], r1 = a.seq_row_off[k + 1];
  r0 = r0 < 0 ? 0 : (r0 > a.n_rows ? a.n_rows : r0);
  r1 = r1 < r0 ? r0 : (r1 > a.n_rows ? a.n_rows : r1);
  const int64_t L = r1 - r0;
  double slr = 0.0, skl = 0.0;
  int bad = 0;
  for (int64_t t = r0 + lane; t < r1; t += 32) {
    const float lp = a.logp[t];
    if (!isfinite(lp)) bad = 1;
    slr += (double)lp - (double)a.old_logp[t];
    const float x = a.ref_logp[t] - lp;
    skl += (double)(expm1f(x) - x);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    slr += __shfl_xor_sync(0xffffffffu, slr, o);
    skl += __shfl_xor_sync(0xffffffffu, skl, o);
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
  }
  if (L == 0 || bad) {
    for (int64_t t = r0 + lane; t < r1; t += 32) a.rowsc[t] = make_float4(0.f, 0.f, 0.f, 0.f);
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
    a.seq_loss[k] = -(surr - (double)a.beta * skl / (double)L) * a.inv_nseq;
    if (a.seq_ratio) a.seq_ratio[k] = (float)s;
  }
  const float w = (float)(a.inv_nseq / (double)L);
  const float sa = c ? (float)(s * A) : 0.f;
  for (int64_t t = r0 + lane; t < r1; t += 32) {
    const float x = a.ref_logp[t] - a.logp[t];
    const float coef = w * -(sa + a.beta * expm1f(x));
    const float4 st = a.stats[t];  // {M, S, S without y}
    float neg_scale = -coef / st.y;
    const float dy = coef * (st.z / st.y);
    float shB = -st.x * kLog2e;
    if (fabsf(neg_scale) >= 0x1p-100f) {
      shB += kShiftB;
      neg_scale *= 0x1p-16f;  // 2^-kShiftB
    }
    a.rowsc[t] = make_float4(neg_scale, dy, shB, 0.f);
  }
}

struct DlArgs {
  const float* z;        // [rows][ld]: pass 1's f32 logits
  __nv_bfloat16* dl;     // [rows][ld]
  int64_t ld;            // row stride of both, a multiple of 32
  const float4* rowsc;   // [rows]: {neg_scale, dy, shift, 0} from lmhead_rows_kernel
  const int32_t* y;      // [rows]
  int32_t rows, V, segs;  // segs: tiles of kDlSeg entries per row
};
constexpr int kDlThreads = 256;
constexpr int kDlSeg = kDlThreads * 16;  // two 8-entry vectors per thread and tile

// dlogits from the stored logits, with pass 2's arithmetic on the same f32 values (so the same
// bits as recomputing the tile): d = neg_scale * 2^(z log2(e) + shift), dy at v = y, 0 for v >= V.
// A persistent grid over (row, 4096-entry segment) tiles; each thread reads two 32-byte pieces of
// logits and writes two 16-byte pieces of dlogits, all streaming.
__global__ void __launch_bounds__(kDlThreads) lmhead_dlogits_kernel(const DlArgs a) {
  if (!GRPO_DCHECK(a.ld % 8 == 0 && (int64_t)a.segs * kDlSeg >= a.ld)) return;
  const int64_t n_tiles = (int64_t)a.rows * a.segs;
  for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int64_t row = tile / a.segs;
    const int seg = (int)(tile - row * a.segs);
    const float4 sc = a.rowsc[row];
    const int yv = a.y[row];
    const float* zr = a.z + row * a.ld;
    __nv_bfloat16* dr = a.dl + row * a.ld;
    float4 v[4];
    int e0[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      e0[u] = seg * kDlSeg + u * (kDlThreads * 8) + (int)threadIdx.x * 8;
      if (e0[u] < a.ld) {  // ld is a multiple of 8: the whole vector is inside the row
        v[2 * u] = __ldcs(reinterpret_cast<const float4*>(zr + e0[u]));
        v[2 * u + 1] = __ldcs(reinterpret_cast<const float4*>(zr + e0[u]) + 1);
      }
    }
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      if (e0[u] >= a.ld) continue;
      const float zz[8] = {v[2 * u].x,     v[2 * u].y,     v[2 * u].z,     v[2 * u].w,
                           v[2 * u + 1].x, v[2 * u + 1].y, v[2 * u + 1].z, v[2 * u + 1].w};
      uint32_t pk[4];
#pragma unroll
      for (int k = 0; k < 8; k += 2) {
        float d0 = sc.x * ex2(fmaf(zz[k], kLog2e, sc.z));
        float d1 = sc.x * ex2(fmaf(zz[k + 1], kLog2e, sc.z));
        if (e0[u] + k == yv) d0 = sc.y;
        if (e0[u] + k + 1 == yv) d1 = sc.y;
        if (e0[u] + k >= a.V) d0 = 0.f;
        if (e0[u] + k + 1 >= a.V) d1 = 0.f;
        pk[k / 2] = pack_bf16x2(make_float2(d0, d1));
      }
      __stcs(reinterpret_cast<uint4*>(dr + e0[u]), make_uint4(pk[0], pk[1], pk[2], pk[3]));
    }
  }
}

// Kept rows gathered into a dense block: hidden row src = row_index[t] (16-byte vectors, one CTA
// per row) and its y, old_logp, ref_logp.
__global__ void __launch_bounds__(128) lmhead_gather_kernel(
    const uint4* __restrict__ hidden, int64_t stride_vec, const int64_t* __restrict__ row_index,
    int32_t n_rows, int32_t row_vec, const int32_t* __restrict__ y, const float* __restrict__ old,
    const float* __restrict__ ref, uint4* __restrict__ out, int32_t* __restrict__ y_out,
    float* __restrict__ old_out, float* __restrict__ ref_out) {
  for (int t = blockIdx.x; t < n_rows; t += gridDim.x) {
    const int64_t src = row_index[t];
    if (!GRPO_DCHECK(src >= 0)) continue;
    const uint4* in = hidden + src * stride_vec;
    uint4* o = out + (int64_t)t * row_vec;
    for (int k = threadIdx.x; k < row_vec; k += blockDim.x) o[k] = in[k];
    if (threadIdx.x == 0) {
      y_out[t] = y[src];
      if (old) old_out[t] = old[src];
      if (ref) ref_out[t] = ref[src];
    }
  }
}

// ---- host side ---------------------------------------------------------------------------------

// 2-D bf16 tensor map over rows x cols (row stride `stride` elements), box 64 x box_rows,
// 128-byte swizzle, zero fill outside the tensor.
bool make_map(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int64_t stride,
              uint32_t box_rows) {
  return tc::make_map_bf16(m, base, rows, cols, stride, box_rows);
}

int sm_count() { return tc::sm_count(); }

struct Grid {
  int R, J, grid;
};
// Launch settings of this process (grpo_lmhead_tune): prefetch distance, row lanes (0 = chosen).
// Atomic: another thread may change them while a call reads them.
std::atomic<int> g_prefetch{0};
std::atomic<int> g_row_lanes{0};
// 1: the token loss recomputes the logits in pass 2 instead of storing them in pass 1.
std::atomic<int> g_recompute{0};

// R pair lanes x J vocabulary lanes, one CTA per SM at most.  The weight is read from DRAM about
// once per group of R row-block pairs, so R stays in [4, 8] (all pairs when there are fewer);
// within that, each CTA does ceil(n_pairs / R) pairs x ceil(n_vt / J) tiles while the average is
// n_pairs * n_vt / grid, and R maximises the busy fraction; a smaller R must gain more than 2%
// (fewer row blocks per group means more weight traffic)
//   (n_pairs / (ceil(n_pairs/R) R)) * (n_vt / (ceil(n_vt/J) J)) * (R J / n_sm).
Grid plan(int64_t rows, int V, int n_sm) {
  const int n_rb = (int)((rows + 2 * BM - 1) / (2 * BM));  // row-block pairs
  const int n_vt = (V + BN - 1) / BN;
  Grid best = {1, 1, 1};
  double best_u = -1.0;
  const int lanes = g_row_lanes.load(std::memory_order_relaxed);
  const int r_hi = lanes > 0 ? lanes : kRowLanes;
  const int r_lo = lanes > 0 ? lanes : std::min(kRowLanes, std::max(1, std::min(n_rb, 4)));
  for (int R = r_hi; R >= r_lo; --R) {
    const int Rr = std::max(1, std::min(n_rb, R));
    const int J = std::max(1, std::min({n_vt, std::max(1, n_sm / Rr), kMaxJ}));
    const double groups = (double)((n_rb + Rr - 1) / Rr);
    const double per_cta_tiles = (double)((n_vt + J - 1) / J);
    const double u = ((double)n_rb / (groups * Rr)) * ((double)n_vt / (per_cta_tiles * J)) *
                     ((double)(Rr * J) / (double)std::max(n_sm, 1));
    if (u > best_u * 1.02) {  // visited from the largest R: within 2%, the larger R wins
      best_u = u;
      best = {Rr, J, Rr * J};
    }
  }
  return best;
}

grpo_status launch_tiles(bool bwd, const CUtensorMap& mh, const CUtensorMap& mw,
                         const TileArgs& a, int grid, cudaStream_t s, const char* who) {
  // The shared-memory limit is a per-device function attribute: set it once on each device.
  static std::mutex mu;
  static uint64_t done = 0;  // bit d: set on device d
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: cudaGetDevice: %s", who, cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return fail(GRPO_ERR_UNSUPPORTED, "%s: device %d beyond 64", who, dev);
  {
    std::lock_guard<std::mutex> lk(mu);
    if (!((done >> dev) & 1u)) {
      e = cudaFuncSetAttribute(lmhead_tile_kernel<false>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(lmhead_tile_kernel<true>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
      if (e != cudaSuccess)
        return fail(GRPO_ERR_CUDA, "%s: cudaFuncSetAttribute: %s", who, cudaGetErrorString(e));
      done |= uint64_t(1) << dev;
    }
  }
  if (bwd)
    lmhead_tile_kernel<true><<<grid, kThreads, kSmemBytes, s>>>(mh, mw, a);
  else
    lmhead_tile_kernel<false><<<grid, kThreads, kSmemBytes, s>>>(mh, mw, a);
  count_launches(1);
  return check_launch(who);
}

int64_t padded_v(int32_t V) { return (int64_t)align_up((size_t)V, 32); }

// Rows per chunk.  The default splits the rows into as few chunks as the 4 GiB of bf16 dlogits
// allow, of equal size (a multiple of 128): a short last chunk would leave most of the products'
// tiles and pass 1's row-block pairs idle (at V = 152064, 16384 rows as 14080 + 2304 ran the call
// at 1524 TFLOP/s where V = 128256's single chunk ran at 1718).
int64_t chunk_of(int64_t n_rows, int32_t V, int64_t chunk_rows) {
  int64_t c = chunk_rows;
  if (c <= 0) {
    const int64_t most = std::max<int64_t>(BM, kDefaultChunkBytes / (padded_v(V) * 2) / BM * BM);
    const int64_t n = std::max<int64_t>(1, (n_rows + most - 1) / most);
    c = (n_rows + n - 1) / n;
  }
  c = (c + BM - 1) / BM * BM;
  return std::max<int64_t>(BM, std::min<int64_t>(c, (n_rows + BM - 1) / BM * BM));
}

// Workspace of the backward products' split K (gemm_plan): the larger of the two products' f32
// partials for the full chunk and for the last, shorter one.  Without a device (a size query on
// a machine with no GPU) the plan assumes 152 SMs; a launch that finds less room runs unsplit.
size_t gemm_partial_bytes(int64_t n_rows, int32_t V, int32_t D, int64_t chunk) {
  int n_sm = sm_count();
  if (n_sm <= 0) n_sm = 152;
  size_t most = 0;
  const int64_t last = n_rows % chunk;
  for (int64_t rows : {std::min(chunk, n_rows), last}) {
    if (rows <= 0) continue;
    most = std::max(most, gemm_plan(rows, D, V, n_sm).partial_bytes);  // dh
    most = std::max(most, gemm_plan(V, D, rows, n_sm).partial_bytes);  // dW
  }
  return most;
}

struct WsLayout {
  size_t part, zy, rowsc, row_loss, stats, seq_loss, z, dl, gpart, hid, ys, olds, refs, total;
};
// loss: the backward buffers; n_seqs >= 0: GSPO's statistics and sequence terms instead of the
// per-row loss terms; store_z: a chunk of f32 logits.
WsLayout ws_layout(int64_t n_rows, int32_t V, int32_t D, int64_t chunk, bool own_dl, bool gather,
                   bool loss, int64_t n_seqs = -1, bool store_z = false) {
  WsLayout w;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  const size_t n = (size_t)std::max<int64_t>(n_rows, 1);
  w.part = take(n * (size_t)((V + BN - 1) / BN) * sizeof(float2));
  w.zy = take(n * sizeof(float));
  w.rowsc = take(loss ? n * sizeof(float4) : 0);
  w.row_loss = take(loss && n_seqs < 0 ? n * sizeof(double) : 0);
  w.stats = take(n_seqs >= 0 ? n * sizeof(float4) : 0);
  w.seq_loss = take(n_seqs >= 0 ? (size_t)std::max<int64_t>(n_seqs, 1) * sizeof(double) : 0);
  w.z = take(loss && store_z ? (size_t)chunk * padded_v(V) * 4 : 0);
  w.dl = take(loss && own_dl ? (size_t)chunk * padded_v(V) * 2 : 0);
  w.gpart = take(loss && n_rows > 0 ? gemm_partial_bytes(n_rows, V, D, chunk) : 0);
  w.hid = take(gather ? n * (size_t)D * 2 : 0);
  w.ys = take(gather ? n * 4 : 0);
  w.olds = take(gather ? n * 4 : 0);
  w.refs = take(gather ? n * 4 : 0);
  w.total = o;
  return w;
}

}  // namespace
}  // namespace fastrl

using namespace fastrl;

namespace {

// Shared front of the entries: the optional gather of the rows, the tensor maps, the pass-1
// arguments common to every launch and, with run_pass1, pass 1 (softmax statistics) over every
// row.  Returns the maps and the row arrays in use.
struct Front {
  CUtensorMap mh, mw;
  const void* hid;
  int64_t hstride;
  const int32_t* y;
  const float* old_logp;
  const float* ref_logp;
  int n_sm;
  TileArgs ta;
};

// Pass 1 over rows [c0, c0 + rows): per-tile partial sums and z_y of those rows and, with z, the
// f32 logits of the first z_rows of them (z row t - c0; z_rows < 0: all).
grpo_status launch_pass1(const Front& f, int64_t c0, int64_t rows, float* z, cudaStream_t s,
                         const char* who, int64_t z_rows = -1) {
  const Grid g = plan(rows, f.ta.V, f.n_sm);
  TileArgs ta = f.ta;
  ta.rows = (int32_t)rows;
  ta.row0 = (int32_t)c0;
  ta.n_rb = (int32_t)((rows + BM - 1) / BM);
  ta.R = g.R;
  ta.J = g.J;
  ta.y = f.y + c0;
  ta.part = f.ta.part + c0 * f.ta.n_vt;
  ta.zy = f.ta.zy + c0;
  ta.z = z;
  ta.ldz = padded_v(f.ta.V);
  ta.z_rows = (int32_t)(z_rows < 0 ? rows : std::min(z_rows, rows));
  return launch_tiles(false, f.mh, f.mw, ta, g.grid, s, who);
}

grpo_status check_shape(const char* who, int64_t n_rows, int32_t V, int32_t D,
                        int64_t hidden_stride) {
  if (n_rows < 0 || n_rows >= (int64_t)1 << 31)
    return fail(GRPO_ERR_INVALID_ARG, "%s: n_rows %lld outside [0, 2^31)", who, (long long)n_rows);
  if (V < 1 || D < 8 || D % 8 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: need V >= 1 and D a positive multiple of 8 (V=%d D=%d)",
                who, V, D);
  if (hidden_stride < D || hidden_stride % 8 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: hidden_stride %lld must be >= D and a multiple of 8",
                who, (long long)hidden_stride);
  return GRPO_OK;
}

grpo_status front(const char* who, const void* hidden, int64_t hidden_stride,
                  const int64_t* row_index, int64_t n_rows, const void* weight, int32_t V,
                  int32_t D, const int32_t* y, const float* old_logp, const float* ref_logp,
                  int32_t* status, char* wsb, const WsLayout& L, bool run_pass1, cudaStream_t s,
                  Front* f) {
  grpo_status st;
  f->n_sm = sm_count();
  if (f->n_sm <= 0) return fail(GRPO_ERR_CUDA, "%s: no CUDA device", who);
  f->hid = hidden;
  f->hstride = hidden_stride;
  f->y = y;
  f->old_logp = old_logp;
  f->ref_logp = ref_logp;
  if (row_index) {  // rows taken through row_index are first gathered into a dense block
    __nv_bfloat16* g_hid = reinterpret_cast<__nv_bfloat16*>(wsb + L.hid);
    int32_t* g_y = reinterpret_cast<int32_t*>(wsb + L.ys);
    float* g_old = old_logp ? reinterpret_cast<float*>(wsb + L.olds) : nullptr;
    float* g_ref = ref_logp ? reinterpret_cast<float*>(wsb + L.refs) : nullptr;
    const int blocks = (int)std::min<int64_t>(n_rows, (int64_t)f->n_sm * 16);
    lmhead_gather_kernel<<<blocks, 128, 0, s>>>(
        static_cast<const uint4*>(hidden), hidden_stride / 8, row_index, (int32_t)n_rows, D / 8, y,
        old_logp, ref_logp, reinterpret_cast<uint4*>(g_hid), g_y, g_old, g_ref);
    count_launches(1);
    if ((st = check_launch(who)) != GRPO_OK) return st;
    f->hid = g_hid;
    f->hstride = D;
    f->y = g_y;
    f->old_logp = g_old;
    f->ref_logp = g_ref;
  }
  if (!make_map(&f->mh, f->hid, n_rows, D, f->hstride, BM) || !make_map(&f->mw, weight, V, D, D, BN))
    return fail(GRPO_ERR_CUDA, "%s: cuTensorMapEncodeTiled failed", who);
  TileArgs& ta = f->ta;
  ta = TileArgs{};
  ta.V = V;
  ta.nK = (D + BK - 1) / BK;
  ta.n_vt = (V + BN - 1) / BN;
  ta.prefetch = g_prefetch.load(std::memory_order_relaxed);
  ta.y = f->y;
  ta.part = reinterpret_cast<float2*>(wsb + L.part);
  ta.zy = reinterpret_cast<float*>(wsb + L.zy);
  ta.status = status;
  return run_pass1 ? launch_pass1(*f, 0, n_rows, nullptr, s, who) : GRPO_OK;
}

// Eqs. 1-3 per row for rows [c0, c0 + rows) (ra's row arrays point at row 0).
grpo_status launch_rows(RowArgs ra, int64_t c0, int64_t rows, cudaStream_t s, const char* who) {
  ra.rows = (int32_t)rows;
  ra.part += c0 * ra.n_vt;
  ra.zy += c0;
  ra.y += c0;
  if (ra.old_logp) ra.old_logp += c0;
  if (ra.ref_logp) ra.ref_logp += c0;
  if (ra.row_rollout) ra.row_rollout += c0;
  if (ra.logp_out) ra.logp_out += c0;
  if (ra.row_loss) ra.row_loss += c0;
  if (ra.rowsc) ra.rowsc += c0;
  if (ra.stats) ra.stats += c0;
  lmhead_rows_kernel<<<(unsigned)((rows + kRowWarps - 1) / kRowWarps), kRowWarps * 32, 0, s>>>(ra);
  count_launches(1);
  return check_launch(who);
}

// dlogits of `rows` rows from their stored f32 logits z (row stride padded_v(V)) and scalars.
grpo_status launch_dlogits(const float* z, __nv_bfloat16* dl, const float4* rowsc,
                           const int32_t* y, int64_t rows, int32_t V, int n_sm, cudaStream_t s,
                           const char* who) {
  DlArgs da = {};
  da.z = z;
  da.dl = dl;
  da.ld = padded_v(V);
  da.rowsc = rowsc;
  da.y = y;
  da.rows = (int32_t)rows;
  da.V = V;
  da.segs = (int)((da.ld + kDlSeg - 1) / kDlSeg);
  const int64_t tiles = rows * da.segs;
  const unsigned grid = (unsigned)std::min<int64_t>(tiles, (int64_t)n_sm * 8);
  lmhead_dlogits_kernel<<<grid, kDlThreads, 0, s>>>(da);
  count_launches(1);
  return check_launch(who);
}

// dhidden[c0 : c0 + rows] = dl * W and dW (+)= dl^T * h[c0 : c0 + rows] for one chunk of dlogits.
grpo_status chunk_products(const char* who, const Front& f, int64_t c0, int64_t rows, int32_t V,
                           int32_t D, const void* weight, const __nv_bfloat16* dl, void* dhidden,
                           int32_t dhidden_dtype, float* dweight, bool acc, float* gpart,
                           size_t gpart_bytes, cudaStream_t s) {
  grpo_status st;
  const int64_t ldd = padded_v(V);
  const size_t dh_elem = dhidden_dtype == GRPO_DTYPE_BF16 ? 2 : 4;
  // dh: A = dl [rows][V] (K-major), B = W [V][D]
  if ((st = gemm_bf16(who, false, dl, ldd, weight, D, rows, D, V,
                      static_cast<char*>(dhidden) + c0 * D * dh_elem, D, dhidden_dtype, false,
                      gpart, gpart_bytes, f.ta.status, s)) != GRPO_OK)
    return st;
  // dW: A = dl^T, stored [rows][V] (M-major), B = h [rows][D]
  return gemm_bf16(who, true, dl, ldd, static_cast<const char*>(f.hid) + c0 * f.hstride * 2,
                   f.hstride, V, D, rows, dweight, D, GRPO_DTYPE_F32, acc, gpart, gpart_bytes,
                   f.ta.status, s);
}

// The dlogits of each chunk (pass 2, or with z0 the first chunk from its logits stored by pass
// 1) and the two products, chunk by chunk, from each row's gradient scalars (rowsc).
grpo_status backward(const char* who, const Front& f, const float4* rowsc, int64_t n_rows,
                     int32_t V, int32_t D, const void* weight, void* dhidden,
                     int32_t dhidden_dtype, float* dweight, int32_t accumulate_dweight,
                     void* dlogits_out, __nv_bfloat16* dl_buf, int64_t chunk, float* gpart,
                     size_t gpart_bytes, cudaStream_t s, const float* z0 = nullptr) {
  grpo_status st;
  const int64_t ldd = padded_v(V);
  for (int64_t c0 = 0; c0 < n_rows; c0 += chunk) {
    const int64_t rows = std::min(chunk, n_rows - c0);
    __nv_bfloat16* dl = dlogits_out ? dl_buf + c0 * ldd : dl_buf;
    if (c0 == 0 && z0 != nullptr) {
      if ((st = launch_dlogits(z0, dl, rowsc, f.y, rows, V, f.n_sm, s, who)) != GRPO_OK) return st;
      if ((st = chunk_products(who, f, c0, rows, V, D, weight, dl, dhidden, dhidden_dtype,
                               dweight, accumulate_dweight != 0, gpart, gpart_bytes, s)) != GRPO_OK)
        return st;
      continue;
    }
    const Grid g2 = plan(rows, V, f.n_sm);
    TileArgs tb = f.ta;
    tb.rows = (int32_t)rows;
    tb.row0 = (int32_t)c0;
    tb.n_rb = (int32_t)((rows + BM - 1) / BM);
    tb.R = g2.R;
    tb.J = g2.J;
    tb.y = f.y + c0;
    tb.part = nullptr;
    tb.zy = nullptr;
    tb.rowsc = rowsc + c0;
    tb.dl = dl;
    tb.ldd = ldd;
    if ((st = launch_tiles(true, f.mh, f.mw, tb, g2.grid, s, who)) != GRPO_OK) return st;
    if ((st = chunk_products(who, f, c0, rows, V, D, weight, dl, dhidden, dhidden_dtype, dweight,
                             !(c0 == 0 && !accumulate_dweight), gpart, gpart_bytes, s)) != GRPO_OK)
      return st;
  }
  return GRPO_OK;
}

}  // namespace

extern "C" grpo_status grpo_lmhead_tune(int32_t prefetch, int32_t row_lanes,
                                        int32_t recompute_logits) {
  clear_error();
  if (prefetch < 0 || prefetch > 64 || row_lanes < 0 || row_lanes > kRowLanes ||
      (recompute_logits != 0 && recompute_logits != 1))
    return fail(GRPO_ERR_INVALID_ARG,
                "grpo_lmhead_tune: prefetch in [0, 64], row_lanes in [0, %d], recompute_logits 0 or 1",
                kRowLanes);
  g_prefetch.store(prefetch, std::memory_order_relaxed);
  g_row_lanes.store(row_lanes, std::memory_order_relaxed);
  g_recompute.store(recompute_logits, std::memory_order_relaxed);
  return GRPO_OK;
}

extern "C" int64_t grpo_lmhead_dlogits_stride(int32_t V) { return V >= 1 ? padded_v(V) : 0; }

extern "C" grpo_status grpo_lmhead_logp_fwd(const void* hidden, int64_t hidden_stride,
                                            const int64_t* row_index, int64_t n_rows,
                                            const void* weight, int32_t V, int32_t D,
                                            const int32_t* y, float* logp_out, int32_t* status,
                                            void* ws, size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_lmhead_logp_fwd");
  clear_error();
  const char* who = "grpo_lmhead_logp_fwd";
  grpo_status st = check_shape(who, n_rows, V, D, hidden_stride);
  if (st != GRPO_OK) return st;
  const WsLayout L = ws_layout(n_rows, V, D, 0, false, row_index != nullptr, false);
  bool query_only = false;
  if ((st = workspace_check(ws, ws_bytes, L.total, who, &query_only)) != GRPO_OK || query_only)
    return st;
  if (n_rows == 0) return GRPO_OK;
  if (!hidden || !weight || !y || !logp_out)
    return fail(GRPO_ERR_INVALID_ARG, "%s: a required pointer is NULL", who);
  if (((uintptr_t)hidden | (uintptr_t)weight) % 16 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: hidden and weight must be 16-byte aligned", who);
  cudaStream_t s = as_stream(stream);
  char* wsb = static_cast<char*>(ws);
  Front f;
  if ((st = front(who, hidden, hidden_stride, row_index, n_rows, weight, V, D, y, nullptr, nullptr,
                  status, wsb, L, true, s, &f)) != GRPO_OK)
    return st;
  RowArgs ra = {};
  ra.n_vt = f.ta.n_vt;
  ra.V = V;
  ra.part = f.ta.part;
  ra.zy = f.ta.zy;
  ra.y = f.y;
  ra.logp_out = logp_out;
  ra.status = status;
  ra.mode = 1;
  return launch_rows(ra, 0, n_rows, s, who);
}

extern "C" grpo_status grpo_lmhead_loss_fwd_bwd(
    const void* hidden, int64_t hidden_stride, const int64_t* row_index, int64_t n_rows,
    const void* weight, int32_t V, int32_t D, const int32_t* y, const float* old_logp,
    const float* ref_logp, const float* adv, const int32_t* row_rollout, float eps_low,
    float eps_high, float beta, int32_t agg_mode, int64_t denom_tokens, const int64_t* seq_off,
    int64_t n_seq, void* dhidden, int32_t dhidden_dtype, float* dweight,
    int32_t accumulate_dweight, void* dlogits_out, float* logp_out, double* row_loss_out,
    double* loss_out, int32_t* status, int64_t chunk_rows, void* ws, size_t* ws_bytes,
    grpo_stream_t stream) {
  GRPO_TRACE("grpo_lmhead_loss_fwd_bwd");
  clear_error();
  const char* who = "grpo_lmhead_loss_fwd_bwd";
  grpo_status st = check_shape(who, n_rows, V, D, hidden_stride);
  if (st != GRPO_OK) return st;
  if (agg_mode != 0 && agg_mode != 1)
    return fail(GRPO_ERR_INVALID_ARG, "%s: agg_mode must be 0 or 1", who);
  if (agg_mode == 0 && denom_tokens <= 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: denom_tokens must be positive", who);
  if (agg_mode == 1 && (seq_off == nullptr || n_seq <= 0))
    return fail(GRPO_ERR_INVALID_ARG, "%s: agg_mode 1 needs seq_off and n_seq > 0", who);
  if (dhidden_dtype != GRPO_DTYPE_BF16 && dhidden_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: dhidden_dtype must be BF16 or F32", who);
  if (!(eps_low >= 0.f && eps_low < 1.f && eps_high >= 0.f && beta >= 0.f && eps_high < INFINITY &&
        beta < INFINITY))
    return fail(GRPO_ERR_INVALID_ARG, "%s: need 0 <= eps_low < 1, finite eps_high, beta >= 0", who);

  const bool store_z = g_recompute.load(std::memory_order_relaxed) == 0;
  const int64_t chunk = chunk_of(n_rows, V, chunk_rows);
  const WsLayout L = ws_layout(n_rows, V, D, chunk, dlogits_out == nullptr, row_index != nullptr,
                               true, -1, store_z);
  bool query_only = false;
  if ((st = workspace_check(ws, ws_bytes, L.total, who, &query_only)) != GRPO_OK || query_only)
    return st;

  if (!weight || !loss_out || !dweight ||
      (n_rows > 0 && (!hidden || !y || !old_logp || !ref_logp || !adv || !row_rollout || !dhidden)))
    return fail(GRPO_ERR_INVALID_ARG, "%s: a required pointer is NULL", who);
  if (((uintptr_t)hidden | (uintptr_t)weight | (uintptr_t)dlogits_out) % 16 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: hidden, weight and dlogits_out must be 16-byte aligned",
                who);
  cudaStream_t s = as_stream(stream);
  char* wsb = static_cast<char*>(ws);
  float4* rowsc = reinterpret_cast<float4*>(wsb + L.rowsc);
  double* row_loss = row_loss_out ? row_loss_out : reinterpret_cast<double*>(wsb + L.row_loss);
  __nv_bfloat16* dl_buf = dlogits_out ? static_cast<__nv_bfloat16*>(dlogits_out)
                                      : reinterpret_cast<__nv_bfloat16*>(wsb + L.dl);
  float* gpart = reinterpret_cast<float*>(wsb + L.gpart);
  const size_t gpart_bytes = L.hid - L.gpart;

  if (n_rows == 0) {
    cudaError_t e = cudaMemsetAsync(loss_out, 0, sizeof(double), s);
    if (e == cudaSuccess && !accumulate_dweight)
      e = cudaMemsetAsync(dweight, 0, (size_t)V * D * sizeof(float), s);
    if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
    return GRPO_OK;
  }

  // Gather (with row_index); with the logits recomputed, pass 1 over every row.
  Front f;
  if ((st = front(who, hidden, hidden_stride, row_index, n_rows, weight, V, D, y, old_logp,
                  ref_logp, status, wsb, L, !store_z, s, &f)) != GRPO_OK)
    return st;

  // Row scalars (Eqs. 1-3).
  RowArgs ra = {};
  ra.n_vt = f.ta.n_vt;
  ra.V = V;
  ra.part = f.ta.part;
  ra.zy = f.ta.zy;
  ra.y = f.y;
  ra.old_logp = f.old_logp;
  ra.ref_logp = f.ref_logp;
  ra.adv = adv;
  ra.row_rollout = row_rollout;
  ra.seq_off = seq_off;
  ra.beta = beta;
  // Clip bounds as the fused loss uses them: rho < lo_up <=> rho < 1 - eps_low in exact arithmetic.
  const double lo = 1.0 - (double)eps_low, hi = 1.0 + (double)eps_high;
  ra.lo_rn = (float)lo;
  ra.hi_rn = (float)hi;
  ra.lo_up = ((double)ra.lo_rn < lo) ? std::nextafter(ra.lo_rn, INFINITY) : ra.lo_rn;
  ra.hi_dn = ((double)ra.hi_rn > hi) ? std::nextafter(ra.hi_rn, -INFINITY) : ra.hi_rn;
  ra.agg_mode = agg_mode;
  ra.inv_denom = agg_mode == 0 ? 1.0 / (double)denom_tokens : 0.0;
  ra.inv_denom_f = (float)ra.inv_denom;
  ra.inv_nseq_f = agg_mode == 1 ? (float)(1.0 / (double)n_seq) : 0.f;
  ra.logp_out = logp_out;
  ra.row_loss = row_loss;
  ra.rowsc = rowsc;
  ra.status = status;
  if (!store_z) {  // pass 2 recomputes the tiles of each chunk
    if ((st = launch_rows(ra, 0, n_rows, s, who)) != GRPO_OK) return st;
    if ((st = launch_sum_rows(row_loss, n_rows, nullptr, loss_out, s, who)) != GRPO_OK) return st;
    return backward(who, f, rowsc, n_rows, V, D, weight, dhidden, dhidden_dtype, dweight,
                    accumulate_dweight, dlogits_out, dl_buf, chunk, gpart, gpart_bytes, s);
  }
  // Chunk by chunk: pass 1 stores the chunk's f32 logits, the row scalars follow, dlogits are
  // formed from the stored logits by a streaming pass, then the two products.
  float* zbuf = reinterpret_cast<float*>(wsb + L.z);
  const int64_t ldd = padded_v(V);
  for (int64_t c0 = 0; c0 < n_rows; c0 += chunk) {
    const int64_t rows = std::min(chunk, n_rows - c0);
    if ((st = launch_pass1(f, c0, rows, zbuf, s, who)) != GRPO_OK) return st;
    if ((st = launch_rows(ra, c0, rows, s, who)) != GRPO_OK) return st;
    __nv_bfloat16* dl = dlogits_out ? dl_buf + c0 * ldd : dl_buf;
    if ((st = launch_dlogits(zbuf, dl, rowsc + c0, f.y + c0, rows, V, f.n_sm, s, who)) != GRPO_OK)
      return st;
    if ((st = chunk_products(who, f, c0, rows, V, D, weight, dl, dhidden, dhidden_dtype, dweight,
                             !(c0 == 0 && !accumulate_dweight), gpart, gpart_bytes, s)) != GRPO_OK)
      return st;
  }
  return launch_sum_rows(row_loss, n_rows, nullptr, loss_out, s, who);
}

extern "C" grpo_status grpo_lmhead_gspo_loss_fwd_bwd(
    const void* hidden, int64_t hidden_stride, const int64_t* row_index, int64_t n_rows,
    const void* weight, int32_t V, int32_t D, const int32_t* y, const float* old_logp,
    const float* ref_logp, const float* adv, const int32_t* seq_rollout,
    const int64_t* seq_row_off, int32_t n_seq_rows, int64_t n_seq, float eps_low, float eps_high,
    float beta, void* dhidden, int32_t dhidden_dtype, float* dweight, int32_t accumulate_dweight,
    void* dlogits_out, float* logp_out, float* seq_ratio_out, double* loss_out, int32_t* status,
    int64_t chunk_rows, void* ws, size_t* ws_bytes, grpo_stream_t stream) {
  GRPO_TRACE("grpo_lmhead_gspo_loss_fwd_bwd");
  clear_error();
  const char* who = "grpo_lmhead_gspo_loss_fwd_bwd";
  grpo_status st = check_shape(who, n_rows, V, D, hidden_stride);
  if (st != GRPO_OK) return st;
  if (n_seq_rows < 0 || n_seq <= 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: n_seq_rows = %d, n_seq = %lld", who, n_seq_rows,
                (long long)n_seq);
  if (dhidden_dtype != GRPO_DTYPE_BF16 && dhidden_dtype != GRPO_DTYPE_F32)
    return fail(GRPO_ERR_INVALID_ARG, "%s: dhidden_dtype must be BF16 or F32", who);
  if (!(eps_low >= 0.f && eps_low < 1.f && eps_high >= 0.f && beta >= 0.f && eps_high < INFINITY &&
        beta < INFINITY))
    return fail(GRPO_ERR_INVALID_ARG, "%s: need 0 <= eps_low < 1, finite eps_high, beta >= 0", who);
  const bool store_z = g_recompute.load(std::memory_order_relaxed) == 0;
  const int64_t chunk = chunk_of(n_rows, V, chunk_rows);
  const WsLayout L = ws_layout(n_rows, V, D, chunk, dlogits_out == nullptr, row_index != nullptr,
                               true, n_seq_rows, store_z);
  bool query_only = false;
  if ((st = workspace_check(ws, ws_bytes, L.total, who, &query_only)) != GRPO_OK || query_only)
    return st;
  if (!weight || !loss_out || !dweight || (n_seq_rows > 0 && (!seq_row_off || !seq_rollout || !adv)) ||
      (n_rows > 0 && (!hidden || !y || !old_logp || !ref_logp || !dhidden || !logp_out)))
    return fail(GRPO_ERR_INVALID_ARG, "%s: a required pointer is NULL", who);
  if (((uintptr_t)hidden | (uintptr_t)weight | (uintptr_t)dlogits_out) % 16 != 0)
    return fail(GRPO_ERR_INVALID_ARG, "%s: hidden, weight and dlogits_out must be 16-byte aligned",
                who);
  cudaStream_t s = as_stream(stream);
  char* wsb = static_cast<char*>(ws);
  if (n_rows == 0 || n_seq_rows == 0) {  // no rows or no sequences: loss 0, zero gradients
    cudaError_t e = cudaMemsetAsync(loss_out, 0, sizeof(double), s);
    if (e == cudaSuccess && !accumulate_dweight)
      e = cudaMemsetAsync(dweight, 0, (size_t)V * D * sizeof(float), s);
    if (e == cudaSuccess && n_rows > 0)
      e = cudaMemsetAsync(dhidden, 0,
                          (size_t)n_rows * D * (dhidden_dtype == GRPO_DTYPE_BF16 ? 2 : 4), s);
    if (e == cudaSuccess && dlogits_out && n_rows > 0)
      e = cudaMemsetAsync(dlogits_out, 0, (size_t)n_rows * padded_v(V) * 2, s);
    if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
    return GRPO_OK;
  }
  float4* rowsc = reinterpret_cast<float4*>(wsb + L.rowsc);
  float4* stats = reinterpret_cast<float4*>(wsb + L.stats);
  double* seq_loss = reinterpret_cast<double*>(wsb + L.seq_loss);
  __nv_bfloat16* dl_buf = dlogits_out ? static_cast<__nv_bfloat16*>(dlogits_out)
                                      : reinterpret_cast<__nv_bfloat16*>(wsb + L.dl);

  // Gather (with row_index) and pass 1 over every row, keeping the first chunk's f32 logits.
  Front f;
  if ((st = front(who, hidden, hidden_stride, row_index, n_rows, weight, V, D, y, old_logp,
                  ref_logp, status, wsb, L, false, s, &f)) != GRPO_OK)
    return st;
  float* zbuf = store_z ? reinterpret_cast<float*>(wsb + L.z) : nullptr;
  if ((st = launch_pass1(f, 0, n_rows, zbuf, s, who, chunk)) != GRPO_OK) return st;
  // logp and the softmax statistics of every row.
  RowArgs ra = {};
  ra.n_vt = f.ta.n_vt;
  ra.V = V;
  ra.part = f.ta.part;
  ra.zy = f.ta.zy;
  ra.y = f.y;
  ra.logp_out = logp_out;
  ra.status = status;
  ra.mode = 2;
  ra.stats = stats;
  if ((st = launch_rows(ra, 0, n_rows, s, who)) != GRPO_OK) return st;
  // Rows outside every sequence keep zero gradient scalars.
  cudaError_t e = cudaMemsetAsync(rowsc, 0, (size_t)n_rows * sizeof(float4), s);
  if (e != cudaSuccess) return fail(GRPO_ERR_CUDA, "%s: memset: %s", who, cudaGetErrorString(e));
  // Sequence ratios, loss terms and the rows' gradient scalars.
  SeqArgs sa = {};
  sa.logp = logp_out;
  sa.old_logp = f.old_logp;
  sa.ref_logp = f.ref_logp;
  sa.adv = adv;
  sa.seq_rollout = seq_rollout;
  sa.seq_row_off = seq_row_off;
  sa.n_seq_rows = n_seq_rows;
  sa.n_rows = n_rows;
  sa.lo = 1.0 - (double)eps_low;
  sa.hi = 1.0 + (double)eps_high;
  sa.beta = beta;
  sa.inv_nseq = 1.0 / (double)n_seq;
  sa.stats = stats;
  sa.rowsc = rowsc;
  sa.seq_loss = seq_loss;
  sa.seq_ratio = seq_ratio_out;
  lmhead_gspo_seq_kernel<<<(unsigned)((n_seq_rows + kSeqWarps - 1) / kSeqWarps), kSeqWarps * 32,
                           0, s>>>(sa);
  count_launches(1);
  if ((st = check_launch(who)) != GRPO_OK) return st;
  if ((st = launch_sum_rows(seq_loss, n_seq_rows, nullptr, loss_out, s, who)) != GRPO_OK) return st;
  // the first chunk's dlogits from its kept logits, the others recomputed in pass 2
  return backward(who, f, rowsc, n_rows, V, D, weight, dhidden, dhidden_dtype, dweight,
                  accumulate_dweight, dlogits_out, dl_buf, chunk,
                  reinterpret_cast<float*>(wsb + L.gpart), L.hid - L.gpart, s, zbuf);
}

namespace fastrl {
GRPO_DCHECK_READER(dcheck_read_lmhead)
}  // namespace fastrl
