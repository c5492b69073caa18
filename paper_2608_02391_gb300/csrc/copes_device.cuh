// Device helpers: the word -> normal transform, bf16 packing and streaming accesses.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "copes_internal.h"
#include "normal_coeffs.h"

namespace copes {

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int N>
__device__ __forceinline__ float horner(const float (&c)[N], float v) {
  float r = c[N - 1];
#pragma unroll
  for (int i = N - 2; i >= 0; --i) r = fmaf(r, v, c[i]);
  return r;
}

// Standard normal from one Philox word: eps = Phi^-1(u), u = ((w >> 8) | 1) * 2^-24.
// x = 2u - 1 is formed exactly from the float with exponent 1 and mantissa w >> 9
// (value 2 + (w >> 9) 2^-22):  x = (that - 3) + 2^-23, both steps exact.  Then
// eps = sqrt(2) erfinv(x) = x * R(L), L = log2(1 - x^2), with R a fitted polynomial in L
// on the central range and in sqrt(-L) on the tail (coefficients: normal_coeffs.h).
// R is evaluated relative to its own value, so eps has a small relative error for all x,
// including x near 0 (where L -> 0) and near +-1.
__device__ __forceinline__ float normal_from_word(uint32_t w) {
  const float f = __uint_as_float((w >> 9) | 0x40000000u);
  const float x = __fadd_rn(__fadd_rn(f, -3.0f), 0x1p-23f);
  const float t = __fmaf_rn(-x, x, 1.0f);
  const float L = lg2_approx(t);
  float r;
  if (__builtin_expect(L >= COPES_NORMAL_L_SPLIT, 1)) {
    constexpr float c[COPES_NORMAL_CENTRAL_DEGREE + 1] = COPES_NORMAL_CENTRAL_COEFFS;
    r = horner(c, L);
  } else {
    constexpr float c[COPES_NORMAL_TAIL_DEGREE + 1] = COPES_NORMAL_TAIL_COEFFS;
    r = horner(c, __fadd_rn(sqrt_approx(-L), -COPES_NORMAL_TAIL_SHIFT));
  }
  return __fmul_rn(x, r);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ uint16_t to_bf16_bits(float x) {
  __nv_bfloat16 v = __float2bfloat16_rn(x);
  return *reinterpret_cast<uint16_t *>(&v);
}

// Streaming (evict-first) 16-byte load of read-once data and matching stores.
__device__ __forceinline__ float4 ld_stream_f4(const float *p) {
  return __ldcs(reinterpret_cast<const float4 *>(p));
}
__device__ __forceinline__ void st_stream_f4(float *p, float4 v) {
  __stcs(reinterpret_cast<float4 *>(p), v);
}
__device__ __forceinline__ void st_stream_u2(void *p, uint2 v) {
  __stcs(reinterpret_cast<uint2 *>(p), v);
}

}  // namespace copes
