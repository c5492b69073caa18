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

// The four words of one Philox block: normal_parts for each, with the central polynomial
// evaluated on two packed pairs (central2 holds each coefficient twice, (c, c); the same
// results bit for bit) and a single warp vote for the tail (taken by a warp with
// probability ~6%), so the common path carries no per-normal branch.
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

__device__ __forceinline__ unsigned long long add_f32x2(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long mul_f32x2(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long splat_f32x2(float c) {
  const unsigned long long b = __float_as_uint(c);
  return (b << 32) | b;
}

// The normals of G Philox blocks with a single warp vote for the tail, every step on packed
// fp32 pairs with compile-time coefficients: each block's central polynomial, then, only
// when some lane of the warp holds a word in the tail, the tail polynomial for those words.  x2[i][p] = (x_2p, x_2p+1) and r2[i][p] = (r_2p, r_2p+1) of
// block i, eps = x * r.  Each packed op rounds like its scalar form and x^2 - 1 is the
// exact negative of 1 - x^2 under round-to-nearest, so each eps is normal_from_word of its
// word bit for bit, with one vote for G blocks instead of one per word.
template <int G>
__device__ __forceinline__ void normal_parts_groups_packed(const uint32_t (&w)[G][4],
                                                           unsigned long long (&x2)[G][2],
                                                           unsigned long long (&r2)[G][2]) {
  COPES_UNIT_COEFFS;
  float L[G][4];
  float L_min = 0.0f;
#pragma unroll
  for (int i = 0; i < G; ++i) {
#pragma unroll
    for (int p = 0; p < 2; ++p) {
      const unsigned long long F = pack_f32x2(__uint_as_float((w[i][2 * p] & 0x007FFFFEu) | 0x40000001u),
                                              __uint_as_float((w[i][2 * p + 1] & 0x007FFFFEu) | 0x40000001u));
      x2[i][p] = add_f32x2(F, splat_f32x2(-3.0f));
      float t0, t1;  // x^2 - 1 = -(1 - x^2)
      unpack_f32x2(fma_f32x2(x2[i][p], x2[i][p], splat_f32x2(-1.0f)), t0, t1);
      L[i][2 * p] = lg2_approx(-t0);
      L[i][2 * p + 1] = lg2_approx(-t1);
      L_min = fminf(L_min, fminf(L[i][2 * p], L[i][2 * p + 1]));
      const unsigned long long Lp = pack_f32x2(L[i][2 * p], L[i][2 * p + 1]);
      unsigned long long acc = splat_f32x2(unit_central[COPES_NORMAL_CENTRAL_DEGREE]);
#pragma unroll
      for (int k = COPES_NORMAL_CENTRAL_DEGREE - 1; k >= 0; --k) acc = fma_f32x2(acc, Lp, splat_f32x2(unit_central[k]));
      r2[i][p] = acc;
    }
  }
  if (__any_sync(__activemask(), L_min < COPES_NORMAL_L_SPLIT)) {
#pragma unroll
    for (int i = 0; i < G; ++i)
#pragma unroll
      for (int p = 0; p < 2; ++p) {
        float r0, r1;
        unpack_f32x2(r2[i][p], r0, r1);
        if (L[i][2 * p] < COPES_NORMAL_L_SPLIT) r0 = tail_ratio(unit_tail, L[i][2 * p]);
        if (L[i][2 * p + 1] < COPES_NORMAL_L_SPLIT) r1 = tail_ratio(unit_tail, L[i][2 * p + 1]);
        r2[i][p] = pack_f32x2(r0, r1);
      }
  }
}

// normal_parts4_x2 over G Philox blocks with a single warp vote for the tail: every
// block's x and r = R(L) scaled by the caller's coefficients (central2 as (c, c) pairs),
// then, only when some lane of the warp holds a word in the tail, the tail polynomial for
// those words.  Each result is the same function of its word as in normal_parts4_x2, bit
// for bit, with one vote for G blocks instead of one per block.
template <int G, int NC, int NT>
__device__ __forceinline__ void normal_parts_groups_x2(const uint32_t (&w)[G][4],
                                                       const unsigned long long (&central2)[NC],
                                                       const float (&tail)[NT], float (&x)[G][4],
                                                       float (&r)[G][4]) {
  float L[G][4];
  float L_min = 0.0f;  // L <= 0 for every word
#pragma unroll
  for (int i = 0; i < G; ++i) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      x[i][e] = lattice_x(w[i][e]);
      L[i][e] = lg2_approx(__fmaf_rn(-x[i][e], x[i][e], 1.0f));
      L_min = fminf(L_min, L[i][e]);
    }
#pragma unroll
    for (int p = 0; p < 2; ++p) {
      const unsigned long long Lp = pack_f32x2(L[i][2 * p], L[i][2 * p + 1]);
      unsigned long long acc = central2[NC - 1];
#pragma unroll
      for (int k = NC - 2; k >= 0; --k) acc = fma_f32x2(acc, Lp, central2[k]);
      unpack_f32x2(acc, r[i][2 * p], r[i][2 * p + 1]);
    }
  }
  if (__any_sync(__activemask(), L_min < COPES_NORMAL_L_SPLIT)) {
#pragma unroll
    for (int i = 0; i < G; ++i)
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (L[i][e] < COPES_NORMAL_L_SPLIT) r[i][e] = tail_ratio(tail, L[i][e]);
  }
}

// normal_parts_groups_x2 with every step on packed pairs, as in normal_parts_groups_packed
// but with the caller's scaled coefficients (central2: (c, c) pairs): x2[i][p] and r2[i][p]
// hold words 2p and 2p + 1 of block i, each value normal_parts_groups_x2's bit for bit.
template <int G, int NC, int NT>
__device__ __forceinline__ void normal_parts_groups_x2_packed(const uint32_t (&w)[G][4],
                                                              const unsigned long long (&central2)[NC],
                                                              const float (&tail)[NT],
                                                              unsigned long long (&x2)[G][2],
                                                              unsigned long long (&r2)[G][2]) {
  float L[G][4];
  float L_min = 0.0f;  // L <= 0 for every word
#pragma unroll
  for (int i = 0; i < G; ++i) {
#pragma unroll
    for (int p = 0; p < 2; ++p) {
      const unsigned long long F = pack_f32x2(__uint_as_float((w[i][2 * p] & 0x007FFFFEu) | 0x40000001u),
                                              __uint_as_float((w[i][2 * p + 1] & 0x007FFFFEu) | 0x40000001u));
      x2[i][p] = add_f32x2(F, splat_f32x2(-3.0f));
      float t0, t1;  // x^2 - 1 = -(1 - x^2)
      unpack_f32x2(fma_f32x2(x2[i][p], x2[i][p], splat_f32x2(-1.0f)), t0, t1);
      L[i][2 * p] = lg2_approx(-t0);
      L[i][2 * p + 1] = lg2_approx(-t1);
      L_min = fminf(L_min, fminf(L[i][2 * p], L[i][2 * p + 1]));
      const unsigned long long Lp = pack_f32x2(L[i][2 * p], L[i][2 * p + 1]);
      unsigned long long acc = central2[NC - 1];
#pragma unroll
      for (int k = NC - 2; k >= 0; --k) acc = fma_f32x2(acc, Lp, central2[k]);
      r2[i][p] = acc;
    }
  }
  if (__any_sync(__activemask(), L_min < COPES_NORMAL_L_SPLIT)) {
#pragma unroll
    for (int i = 0; i < G; ++i)
#pragma unroll
      for (int p = 0; p < 2; ++p) {
        float r0, r1;
        unpack_f32x2(r2[i][p], r0, r1);
        if (L[i][2 * p] < COPES_NORMAL_L_SPLIT) r0 = tail_ratio(tail, L[i][2 * p]);
        if (L[i][2 * p + 1] < COPES_NORMAL_L_SPLIT) r1 = tail_ratio(tail, L[i][2 * p + 1]);
        r2[i][p] = pack_f32x2(r0, r1);
      }
  }
}

// Two standard normals from two words (of different Philox blocks), their central
// polynomials evaluated as one packed pair with compile-time coefficients and a single
// warp vote for the tail: bit-identical to two normal_from_word calls.
__device__ __forceinline__ void normal_pair_x2(uint32_t wa, uint32_t wb, float &ea, float &eb) {
  COPES_UNIT_COEFFS;
  const float xa = lattice_x(wa), xb = lattice_x(wb);
  const float La = lg2_approx(__fmaf_rn(-xa, xa, 1.0f));
  const float Lb = lg2_approx(__fmaf_rn(-xb, xb, 1.0f));
  const unsigned long long Lp = pack_f32x2(La, Lb);
  unsigned long long b = __float_as_uint(unit_central[COPES_NORMAL_CENTRAL_DEGREE]);
  unsigned long long acc = (b << 32) | b;
#pragma unroll
  for (int k = COPES_NORMAL_CENTRAL_DEGREE - 1; k >= 0; --k) {
    b = __float_as_uint(unit_central[k]);
    acc = fma_f32x2(acc, Lp, (b << 32) | b);
  }
  float ra, rb;
  unpack_f32x2(acc, ra, rb);
  if (__any_sync(__activemask(), fminf(La, Lb) < COPES_NORMAL_L_SPLIT)) {
    if (La < COPES_NORMAL_L_SPLIT) ra = tail_ratio(unit_tail, La);
    if (Lb < COPES_NORMAL_L_SPLIT) rb = tail_ratio(unit_tail, Lb);
  }
  ea = __fmul_rn(xa, ra);
  eb = __fmul_rn(xb, rb);
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

// ------------------------------------------------------------------------------------
// Gather-list staging: a block's segment of the int64 index list is brought into shared
// memory by TMA 1D bulk copies (cp.async.bulk) in chunks, double-buffered on mbarriers,
// so the next chunk's indices are in flight while the current chunk is processed.
// Every wait is bounded: after kStageWaitLimit polls the block records kErrStageTimeout,
// waits (bounded again) for its own copies, and stops.
constexpr int kStageChunk = 1024;         // indices per chunk (8 KB)
constexpr int kStageWaitLimit = 1 << 22;  // mbarrier polls before giving up

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// One producer arrival announcing `bytes` of transaction, then the bulk copy itself.
__device__ __forceinline__ void stage_copy(uint64_t *bar, void *dst, const void *src, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
  if (bytes)
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// Polls the barrier's phase `parity` at most kStageWaitLimit times; true once complete.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity) {
  for (int it = 0; it < kStageWaitLimit; ++it) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}

// Walks the block's segment [s0, s1) of `index` in chunks staged through shared memory;
// body(const int64_t *chunk_in_smem, int count, uint64_t first_position) runs on every
// chunk with all threads of the block.  A chunk of odd length copies its even prefix by
// TMA (sizes must be multiples of 16 bytes) and its last index from global memory into
// shared memory.  Returns false (after flagging) if a wait timed out.
template <typename Body, typename Flag>
__device__ __forceinline__ bool staged_index_segment(const int64_t *index, uint64_t s0, uint64_t s1,
                                                     int64_t (*buf)[kStageChunk], uint64_t *bar,
                                                     Flag flag, Body body) {
  const int n_chunks = (int)((s1 - s0 + kStageChunk - 1) / kStageChunk);
  auto chunk_count = [&](int c) { return (int)min((uint64_t)kStageChunk, s1 - s0 - (uint64_t)c * kStageChunk); };
  auto issue = [&](int c) {
    const int cnt = chunk_count(c);
    stage_copy(&bar[c & 1], buf[c & 1], index + s0 + (uint64_t)c * kStageChunk, (uint32_t)(cnt & ~1) * 8u);
  };
  if (threadIdx.x == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    issue(0);
    if (n_chunks > 1) issue(1);
  }
  for (int c = 0; c < n_chunks; ++c) {
    const int slot = c & 1;
    const int cnt = chunk_count(c);
    if (!mbar_wait_bounded(&bar[slot], (uint32_t)((c >> 1) & 1))) {
      if (threadIdx.x == 0) flag();
      // the copy into this block's shared memory may still be in flight: wait once more
      mbar_wait_bounded(&bar[slot], (uint32_t)((c >> 1) & 1));
      return false;
    }
    if ((cnt & 1) && threadIdx.x == 0) buf[slot][cnt - 1] = index[s0 + (uint64_t)c * kStageChunk + cnt - 1];
    __syncthreads();
    body((const int64_t *)buf[slot], cnt, s0 + (uint64_t)c * kStageChunk);
    __syncthreads();  // every thread is done reading this slot before it is refilled
    if (threadIdx.x == 0 && c + 2 < n_chunks) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      issue(c + 2);
    }
  }
  return true;
}

}  // namespace copes
