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

// ---- rows that do not start on a 16-byte boundary ---------------------------------------------

// Bytes [off, off + 16) of the 32 bytes lo:hi (lo first, little-endian), 0 <= off < 16: the
// 16-byte vector that starts off bytes into lo, assembled from the two aligned words that hold
// it by 32-bit funnel shifts.
__device__ __forceinline__ uint4 extract16(const uint4& lo, const uint4& hi, int off) {
  const uint32_t sh = (uint32_t)(off & 3) * 8u;
  uint32_t w0, w1, w2, w3, w4;
  switch (off >> 2) {  // the word holding byte off; branches keep the words in registers
    case 0: w0 = lo.x; w1 = lo.y; w2 = lo.z; w3 = lo.w; w4 = hi.x; break;
    case 1: w0 = lo.y; w1 = lo.z; w2 = lo.w; w3 = hi.x; w4 = hi.y; break;
    case 2: w0 = lo.z; w1 = lo.w; w2 = hi.x; w3 = hi.y; w4 = hi.z; break;
    default: w0 = lo.w; w1 = hi.x; w2 = hi.y; w3 = hi.z; w4 = hi.w; break;
  }
  return make_uint4(__funnelshift_r(w0, w1, sh), __funnelshift_r(w1, w2, sh),
                    __funnelshift_r(w2, w3, sh), __funnelshift_r(w3, w4, sh));
}

// extract16 for a word offset known at compile time: bytes [4 Q + sh / 8, 4 Q + sh / 8 + 16) of
// lo:hi, sh in {0, 8, 16, 24} (the byte offset's remainder, in bits), so that a loop over
// vectors of one row keeps only the four funnel shifts.
template <int Q>
__device__ __forceinline__ uint4 extract16_q(const uint4& lo, const uint4& hi, uint32_t sh) {
  const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
  return make_uint4(__funnelshift_r(w[Q], w[Q + 1], sh), __funnelshift_r(w[Q + 1], w[Q + 2], sh),
                    __funnelshift_r(w[Q + 2], w[Q + 3], sh), __funnelshift_r(w[Q + 3], w[Q + 4], sh));
}

// Elements per 16-byte word of the output, and the input bytes they come from.
template <typename InT, typename OutT>
struct OutWord {
  static constexpr int kElems = 16 / (int)sizeof(OutT);
  static constexpr int kPairs = kElems / 2;
  static constexpr int kInBytes = kElems * (int)sizeof(InT);  // 8, 16 or 32
};

// The OutWord<InT, OutT>::kElems inputs that start off bytes into the aligned words w0, w1, w2
// (w1 and w2 are read only when those bytes reach them), as f32 pairs.
template <typename InT, typename OutT>
__device__ __forceinline__ void pairs_from_words(const uint4& w0, const uint4& w1, const uint4& w2,
                                                 int off, float2 (&p)[OutWord<InT, OutT>::kPairs]) {
  constexpr int kIn = OutWord<InT, OutT>::kInBytes;
  if constexpr (kIn == 16) {  // bf16 -> bf16 or f32 -> f32: one input vector
    Fmt<InT>::pairs(off ? extract16(w0, w1, off) : w0, p);
  } else if constexpr (kIn == 8) {  // bf16 -> f32: four bf16 in the low 8 bytes
    const uint4 q = extract16(w0, off > 8 ? w1 : w0, off);
    p[0] = Fmt<__nv_bfloat16>::pair(q.x);
    p[1] = Fmt<__nv_bfloat16>::pair(q.y);
  } else {  // f32 -> bf16: eight f32 from two input vectors
    const uint4 q0 = off ? extract16(w0, w1, off) : w0;
    const uint4 q1 = off ? extract16(w1, w2, off) : w1;
    p[0] = make_float2(__uint_as_float(q0.x), __uint_as_float(q0.y));
    p[1] = make_float2(__uint_as_float(q0.z), __uint_as_float(q0.w));
    p[2] = make_float2(__uint_as_float(q1.x), __uint_as_float(q1.y));
    p[3] = make_float2(__uint_as_float(q1.z), __uint_as_float(q1.w));
  }
}

// Aligned 16-byte words that hold kIn bytes starting off bytes into the first.
__host__ __device__ constexpr int words_for(int off, int in_bytes) { return (off + in_bytes + 15) >> 4; }

// The OutWord<InT, OutT>::kElems inputs of elements [i0, i0 + kElems) of an element-aligned
// array v16 (16-byte words; element 0 at byte 0), as f32 pairs.  Reads only the words that hold
// those bytes, so v16 may end at the last one.
template <typename InT, typename OutT>
__device__ __forceinline__ void pairs_at(const uint4* v16, int i0,
                                         float2 (&p)[OutWord<InT, OutT>::kPairs]) {
  constexpr int kIn = OutWord<InT, OutT>::kInBytes;
  const int b = i0 * (int)sizeof(InT);
  const int idx = b >> 4, off = b & 15;
  const int nw = words_for(off, kIn);
  const uint4 w0 = v16[idx];
  const uint4 w1 = nw > 1 ? v16[idx + 1] : w0;
  const uint4 w2 = nw > 2 ? v16[idx + 2] : w1;
  pairs_from_words<InT, OutT>(w0, w1, w2, off, p);
}

// The same from a row of V elements in global memory that may start anywhere on an element
// boundary: the aligned words holding the bytes are loaded (streaming) when all of them lie
// inside the row, else the elements are loaded one by one.
template <typename InT, typename OutT>
__device__ __forceinline__ void pairs_at_global(const InT* row, int V, int i0,
                                                float2 (&p)[OutWord<InT, OutT>::kPairs]) {
  constexpr int kIn = OutWord<InT, OutT>::kInBytes;
  const int mis = (int)(reinterpret_cast<uintptr_t>(row) & 15u);
  const int b = mis + i0 * (int)sizeof(InT);
  const int idx = b >> 4, off = b & 15;
  const int nw = words_for(off, kIn);
  if ((mis == 0 || idx >= 1) && 16 * (int64_t)(idx + nw) <= (int64_t)V * (int64_t)sizeof(InT) + mis) {
    const uint4* base = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(row) - mis) + idx;
    const uint4 w0 = __ldcs(base);
    const uint4 w1 = nw > 1 ? __ldcs(base + 1) : w0;
    const uint4 w2 = nw > 2 ? __ldcs(base + 2) : w1;
    pairs_from_words<InT, OutT>(w0, w1, w2, off, p);
  } else {
#pragma unroll
    for (int i = 0; i < OutWord<InT, OutT>::kPairs; ++i)
      p[i] = make_float2(Fmt<InT>::load(row + i0 + 2 * i), Fmt<InT>::load(row + i0 + 2 * i + 1));
  }
}

// The 16-byte vector of elements [j kVec, (j + 1) kVec) of a row that starts mis bytes past a
// 16-byte boundary (mis a multiple of the element size, V elements): two aligned loads and
// funnel shifts when both words lie inside the row, else element loads.
template <typename InT>
__device__ __forceinline__ uint4 vec_at_global(const InT* row, int mis, int V, int j) {
  if (mis == 0) return __ldcs(reinterpret_cast<const uint4*>(row) + j);
  const uint4* base = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(row) - mis);
  if (j >= 1 && 16 * (int64_t)(j + 2) <= (int64_t)V * (int64_t)sizeof(InT) + mis)
    return extract16(__ldcs(base + j), __ldcs(base + j + 1), mis);
  uint32_t w[4];
  if constexpr (sizeof(InT) == 2) {
    const uint16_t* e = reinterpret_cast<const uint16_t*>(row) + j * 8;
#pragma unroll
    for (int i = 0; i < 4; ++i) w[i] = (uint32_t)e[2 * i] | ((uint32_t)e[2 * i + 1] << 16);
  } else {
    const uint32_t* e = reinterpret_cast<const uint32_t*>(row) + j * 4;
#pragma unroll
    for (int i = 0; i < 4; ++i) w[i] = e[i];
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

}  // namespace
}  // namespace fastrl
