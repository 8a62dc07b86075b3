// Element-level device helpers shared by the row kernels of libfastrl_grpo (the fused loss, the
// forward-only log-probabilities and GSPO's dlogits pass): base-2 exponentials on the MUFU,
// 16-byte vectors of bf16 or f32 logits unpacked into f32 pairs, and streaming vector stores.
#pragma once

#include <cuda_bf16.h>

#include "common.cuh"

namespace fastrl {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

// 2^x on the MUFU (one instruction); results below 2^-126 flush to zero.  Pass A only loses
// terms 2^126 times smaller than the running maximum; pass B shifts its argument (see
// kShiftB) so that no representable gradient entry is lost.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float2 ex2x2(float2 t) { return make_float2(ex2(t.x), ex2(t.y)); }
// Lane-wise maximum of two bf16 pairs; a NaN operand yields the other operand.
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Pass B evaluates 2^(t + kShiftB) * (scale * 2^-kShiftB) when |scale| >= 2^-100, which moves the
// flush-to-zero point of ex2 below every gradient entry that bf16 or f32 can represent.
constexpr float kShiftB = 16.f;

// ---- element formats: 16-byte vectors of the logits, unpacked into f32 pairs -----------------

template <typename T>
struct Fmt;
template <>
struct Fmt<float> {
  static constexpr int kVec = 4;  // elements per 16 bytes
  static constexpr int kPairs = 2;
  __device__ static void pairs(const uint4& q, float2 (&p)[2]) {
    p[0] = make_float2(__uint_as_float(q.x), __uint_as_float(q.y));
    p[1] = make_float2(__uint_as_float(q.z), __uint_as_float(q.w));
  }
  struct Max {  // running maximum over vectors
    float m = -INFINITY;
    __device__ void add(const uint4& q) {
      m = fmaxf(m, fmaxf(fmaxf(__uint_as_float(q.x), __uint_as_float(q.y)),
                         fmaxf(__uint_as_float(q.z), __uint_as_float(q.w))));
    }
    __device__ float get() const { return m; }
  };
  __device__ static float load(const float* p) { return *p; }
  __device__ static void store(float* p, float v) { *p = v; }
};
template <>
struct Fmt<__nv_bfloat16> {
  static constexpr int kVec = 8;
  static constexpr int kPairs = 4;
  __device__ static float2 pair(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
  }
  __device__ static void pairs(const uint4& q, float2 (&p)[4]) {
    p[0] = pair(q.x);
    p[1] = pair(q.y);
    p[2] = pair(q.z);
    p[3] = pair(q.w);
  }
  struct Max {  // running maximum kept as a bf16 pair: one instruction per two elements
    uint32_t m = 0xFF80FF80u;  // (-inf, -inf)
    __device__ void add(const uint4& q) { m = bmax2(m, bmax2(bmax2(q.x, q.y), bmax2(q.z, q.w))); }
    __device__ float get() const {
      return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
    }
  };
  __device__ static float load(const __nv_bfloat16* p) { return __bfloat162float(*p); }
  __device__ static void store(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }
};

__device__ __forceinline__ uint32_t pack_bf16x2(float2 v) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(v.x, v.y);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Store one vector of results at p (aligned to its width), streaming (evict-first).
template <typename OutT, int kPairs>
__device__ __forceinline__ void store_pairs(OutT* p, const float2 (&d)[kPairs]);
template <>
__device__ __forceinline__ void store_pairs<__nv_bfloat16, 4>(__nv_bfloat16* p, const float2 (&d)[4]) {
  __stcs(reinterpret_cast<uint4*>(p),
         make_uint4(pack_bf16x2(d[0]), pack_bf16x2(d[1]), pack_bf16x2(d[2]), pack_bf16x2(d[3])));
}
template <>
__device__ __forceinline__ void store_pairs<float, 4>(float* p, const float2 (&d)[4]) {
  __stcs(reinterpret_cast<float4*>(p), make_float4(d[0].x, d[0].y, d[1].x, d[1].y));
  __stcs(reinterpret_cast<float4*>(p) + 1, make_float4(d[2].x, d[2].y, d[3].x, d[3].y));
}
template <>
__device__ __forceinline__ void store_pairs<float, 2>(float* p, const float2 (&d)[2]) {
  __stcs(reinterpret_cast<float4*>(p), make_float4(d[0].x, d[0].y, d[1].x, d[1].y));
}
template <>
__device__ __forceinline__ void store_pairs<__nv_bfloat16, 2>(__nv_bfloat16* p, const float2 (&d)[2]) {
  __stcs(reinterpret_cast<uint2*>(p), make_uint2(pack_bf16x2(d[0]), pack_bf16x2(d[1])));
}
template <typename OutT, int kPairs>
__device__ __forceinline__ void store_pairs_scalar(OutT* p, const float2 (&d)[kPairs]) {
#pragma unroll
  for (int i = 0; i < kPairs; ++i) {
    Fmt<OutT>::store(p + 2 * i, d[i].x);
    Fmt<OutT>::store(p + 2 * i + 1, d[i].y);
  }
}

}  // namespace
}  // namespace fastrl
