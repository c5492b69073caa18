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
  // Horner's rule, highest coefficient first
  float r = c[N - 1];
#pragma unroll
  for (int i = N - 2; i >= 0; --i) r = __fmaf_rn(r, v, c[i]);
  return r;
}

// Standard normal from one Philox word w: eps = Phi^-1(u), u = ((w & 0x7FFFFE) | 1) 2^-23.
// OR-ing those bits (made odd) under the exponent of 2 gives the float 2 + m 2^-22 with m
// odd, so x = 2u - 1 = that - 3 is exact in one add.  Then
//   eps = sqrt(2) erfinv(x) = x * R(L),  L = log2(1 - x^2),
// with R a fitted polynomial in L on the central range and in sqrt(-L) - shift on the tail
// (coefficients: normal_coeffs.h).  R is evaluated relative to its own value, so eps has
// a small relative error for every x, including x near 0 (L -> 0) and near +-1.
//
// The parts return x and r = scale * R(L) when given coefficients pre-multiplied by
// scale, so a caller forms scale * eps + b as one fma(r, x, b).
__device__ __forceinline__ float lattice_x(uint32_t w) {
  return __fadd_rn(__uint_as_float((w & 0x007FFFFEu) | 0x40000001u), -3.0f);
}

template <int NT>
__device__ __forceinline__ float tail_ratio(const float (&tail)[NT], float L) {
  return horner(tail, __fadd_rn(sqrt_approx(-L), -COPES_NORMAL_TAIL_SHIFT));
}

// One word.  The tail polynomial runs only when some active lane needs it.
template <int NC, int NT>
__device__ __forceinline__ void normal_parts(uint32_t w, const float (&central)[NC],
                                             const float (&tail)[NT], float &x, float &r) {
  x = lattice_x(w);
  const float L = lg2_approx(__fmaf_rn(-x, x, 1.0f));
  r = horner(central, L);
  const bool in_tail = L < COPES_NORMAL_L_SPLIT;
  if (__any_sync(__activemask(), in_tail)) {
    if (in_tail) r = tail_ratio(tail, L);
  }
}

// The four words of one Philox block with a single warp vote for the tail (taken by a
// warp with probability ~6%), so the common path carries no per-normal branch.
template <int NC, int NT>
__device__ __forceinline__ void normal_parts4(const uint32_t (&w)[4], const float (&central)[NC],
                                              const float (&tail)[NT], float (&x)[4],
                                              float (&r)[4]) {
  float L[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    x[e] = lattice_x(w[e]);
    L[e] = lg2_approx(__fmaf_rn(-x[e], x[e], 1.0f));
    r[e] = horner(central, L[e]);
  }
  const float L_min = fminf(fminf(L[0], L[1]), fminf(L[2], L[3]));
  if (__any_sync(__activemask(), L_min < COPES_NORMAL_L_SPLIT)) {
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (L[e] < COPES_NORMAL_L_SPLIT) r[e] = tail_ratio(tail, L[e]);
  }
}

// Packed fp32 pairs: one fma.rn.f32x2 performs the two lanes' fp32 fmas, each rounded
// exactly as a scalar fma, at half the instruction count.
__device__ __forceinline__ unsigned long long pack_f32x2(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack_f32x2(unsigned long long v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ unsigned long long fma_f32x2(unsigned long long a, unsigned long long b,
                                                        unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// normal_parts4 with the central polynomial evaluated on two pairs of normals; central2
// holds each coefficient twice (c, c).  Same results as normal_parts4, bit for bit.
template <int NC, int NT>
__device__ __forceinline__ void normal_parts4_x2(const uint32_t (&w)[4],
                                                 const unsigned long long (&central2)[NC],
                                                 const float (&tail)[NT], float (&x)[4],
                                                 float (&r)[4]) {
  float L[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    x[e] = lattice_x(w[e]);
    L[e] = lg2_approx(__fmaf_rn(-x[e], x[e], 1.0f));
  }
#pragma unroll
  for (int p = 0; p < 2; ++p) {
    const unsigned long long Lp = pack_f32x2(L[2 * p], L[2 * p + 1]);
    unsigned long long acc = central2[NC - 1];
#pragma unroll
    for (int i = NC - 2; i >= 0; --i) acc = fma_f32x2(acc, Lp, central2[i]);
    unpack_f32x2(acc, r[2 * p], r[2 * p + 1]);
  }
  const float L_min = fminf(fminf(L[0], L[1]), fminf(L[2], L[3]));
  if (__any_sync(__activemask(), L_min < COPES_NORMAL_L_SPLIT)) {
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (L[e] < COPES_NORMAL_L_SPLIT) r[e] = tail_ratio(tail, L[e]);
  }
}

#define COPES_UNIT_COEFFS                                                                     \
  constexpr float unit_central[COPES_NORMAL_CENTRAL_DEGREE + 1] = COPES_NORMAL_CENTRAL_COEFFS; \
  constexpr float unit_tail[COPES_NORMAL_TAIL_DEGREE + 1] = COPES_NORMAL_TAIL_COEFFS

__device__ __forceinline__ float normal_from_word(uint32_t w) {
  COPES_UNIT_COEFFS;
  float x, r;
  normal_parts(w, unit_central, unit_tail, x, r);
  return __fmul_rn(x, r);
}

// eps for the four words of one Philox block.
__device__ __forceinline__ void normals4(const uint32_t (&w)[4], float (&eps)[4]) {
  COPES_UNIT_COEFFS;
  float x[4], r[4];
  normal_parts4(w, unit_central, unit_tail, x, r);
#pragma unroll
  for (int e = 0; e < 4; ++e) eps[e] = __fmul_rn(x[e], r[e]);
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
