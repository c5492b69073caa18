// Elementwise ES kernels: perturb (Eq. 8), restore / context commit (Supp. A.8), the
// fused reward-weighted update (Eq. 6 / Eq. 13) and the synthetic initialiser, over
// TILES subspaces (vectorised, 4-element groups = one Philox counter) and INDICES
// subspaces (gather / scatter through a sorted int64 list).
#include <cuda_bf16.h>

#include "copes_device.cuh"
#include "copes_internal.h"
#include "es_common.cuh"

namespace copes {

__device__ unsigned int g_es_error = 0;

__device__ __forceinline__ void flag_error(unsigned bit) { atomicOr(&g_es_error, bit); }

// ----------------------------------------------------------------- group primitives
// A "group" is the 4 consecutive global indices 4q .. 4q+3, which share Philox counter q.

// Noise for a single index g: the one word of its counter that g uses.
__device__ __forceinline__ float index_noise(uint64_t g, uint32_t tag, uint32_t k0, uint32_t k1) {
  uint32_t x[4];
  const uint64_t q = g >> 2;
  philox4x32_10((uint32_t)q, (uint32_t)(q >> 32), 0u, tag, k0, k1, x);
  const uint32_t s = (uint32_t)g & 3u;
  const uint32_t w = s == 0 ? x[0] : (s == 1 ? x[1] : (s == 2 ? x[2] : x[3]));
  return normal_from_word(w);
}

// ------------------------------------------------------------ perturb / restore / init
template <int OP>
constexpr uint32_t op_tag() { return OP == kOpInit ? COPES_TAG_INIT : COPES_TAG_NOISE; }

// Ops whose values are the context (restore / commit, init) go to the second working
// buffer too; perturbations go to w only.
template <int OP>
constexpr bool writes_context() { return OP == kOpRestore || OP == kOpInit; }

// perturb: v = theta + a eps;  init: v = b + a eps;  restore: v = theta;  perturb pair:
// v = theta + a eps and the partner's vp = theta - a eps.  (q_lo, q_hi) is the group's
// Philox counter g4 >> 2.  Coefficients scaled by -a are the exact negatives of those
// scaled by a, so vp equals, bit for bit, what kOpPerturb computes with scale -a.
template <int OP>
__device__ __forceinline__ void elem_values(const ElemArgs &a, uint32_t q_lo, uint32_t q_hi,
                                            const float th[4], float v[4], float vp[4]) {
  if (OP == kOpRestore) {
#pragma unroll
    for (int e = 0; e < 4; ++e) v[e] = th[e];
  } else {
    uint32_t w[4];
    philox4x32_10_rk(q_lo, q_hi, 0u, op_tag<OP>(), a.rk, w);
    float x[4], r[4];
    normal_parts4_x2(w, a.coeffs.central2, a.coeffs.tail, x, r);  // r = a * R(L)
#pragma unroll
    for (int e = 0; e < 4; ++e) v[e] = __fmaf_rn(r[e], x[e], OP == kOpInit ? a.b : th[e]);
    if (OP == kOpPerturbPair) {
#pragma unroll
      for (int e = 0; e < 4; ++e) vp[e] = __fmaf_rn(-r[e], x[e], th[e]);
    }
  }
}

// One step of the pair perturb over the thread's G groups of an aligned tile whose
// counters are all below 2^32: the G groups' Philox calls first, then their transforms
// with one tail vote (normal_parts_groups_x2), then each group's two members -- the
// values elem_values<kOpPerturbPair> computes, bit for bit.  Groups past the tile's end
// are generated but not stored.
template <typename WT, int G>
__device__ __forceinline__ void pair_perturb_step(const ElemArgs &a, uint64_t b, uint32_t len, uint32_t off,
                                                  uint32_t q0_lo, const float (&th)[G][4]) {
  uint32_t w[G][4];
#pragma unroll
  for (int i = 0; i < G; ++i)
    philox4x32_10_rk(q0_lo + ((off + 4u * kThreads * i) >> 2), 0u, 0u, COPES_TAG_NOISE, a.rk, w[i]);
  float x[G][4], r[G][4];  // r = a * R(L)
  normal_parts_groups_x2<G>(w, a.coeffs.central2, a.coeffs.tail, x, r);
#pragma unroll
  for (int i = 0; i < G; ++i) {
    const uint32_t o = off + 4u * kThreads * i;
    if (o >= len) continue;
    float v[4], vp[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[e] = __fmaf_rn(r[i][e], x[i][e], th[i][e]);
      vp[e] = __fmaf_rn(-r[i][e], x[i][e], th[i][e]);
    }
    WStore<WT>::full(a.w, b + o, v);
    WStore<WT>::full(a.partner, b + o - a.partner_base, vp);
  }
}

// Two antithetic pairs of the group at counter (q_lo, q_hi) (kOpPerturbTwoPairs):
// v[0] = theta + a eps_A, v[1] = theta - a eps_A, v[2] = theta + a eps_B and
// v[3] = theta - a eps_B, each bit for bit what kOpPerturb computes with that noise vector
// and sign (normal_parts_groups_x2 gives normal_parts4_x2's values).
__device__ __forceinline__ void two_pairs_values(const ElemArgs &a, uint32_t q_lo, uint32_t q_hi,
                                                 const float th[4], float (&v)[4][4]) {
  uint32_t w[2][4];
  philox4x32_10_rk(q_lo, q_hi, 0u, COPES_TAG_NOISE, a.rk, w[0]);
  philox4x32_10_rk(q_lo, q_hi, 0u, COPES_TAG_NOISE, a.rk_b, w[1]);
  float x[2][4], r[2][4];  // r = a * R(L)
  normal_parts_groups_x2<2>(w, a.coeffs.central2, a.coeffs.tail, x, r);
#pragma unroll
  for (int s = 0; s < 2; ++s)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[2 * s][e] = __fmaf_rn(r[s][e], x[s][e], th[e]);
      v[2 * s + 1][e] = __fmaf_rn(-r[s][e], x[s][e], th[e]);
    }
}

// The four members' values go to w, copies[0], copies[1] and copies[2].
template <typename WT>
__device__ __forceinline__ void store_two_pairs_full(const ElemArgs &a, uint64_t g, const float (&v)[4][4]) {
  WStore<WT>::full(a.w, g, v[0]);
  WStore<WT>::full(a.copies.p[0], g, v[1]);
  WStore<WT>::full(a.copies.p[1], g, v[2]);
  WStore<WT>::full(a.copies.p[2], g, v[3]);
}

template <typename WT>
__device__ __forceinline__ void store_two_pairs_one(const ElemArgs &a, uint64_t g, const float (&v)[4][4], int k) {
  WStore<WT>::one(a.w, g, v[0][k]);
  WStore<WT>::one(a.copies.p[0], g, v[1][k]);
  WStore<WT>::one(a.copies.p[1], g, v[2][k]);
  WStore<WT>::one(a.copies.p[2], g, v[3][k]);
}

// One step of the two-pairs perturb over the thread's G groups of an aligned tile whose
// counters are all below 2^32: each group's product M0 q is computed once and shared by
// both noise vectors' folded Philox (philox4x32_10_folded, the same words as
// philox4x32_10_rk), the 2G blocks' transforms take one tail vote, and each group's four
// members are formed on packed pairs and stored -- two_pairs_values' results, bit for bit
// (the antithetic member as fma(r, -x, theta): -x is exact).  Groups past the tile's end are
// generated but not stored.
template <typename WT, int G>
__device__ __forceinline__ void two_pairs_step(const ElemArgs &a, uint64_t b, uint32_t len, uint32_t off,
                                               uint32_t q0_lo, const float (&th)[G][4]) {
  uint32_t w[2 * G][4];
#pragma unroll
  for (int i = 0; i < G; ++i) {
    const uint64_t m = (uint64_t)kPhiloxM0 * (q0_lo + ((off + 4u * kThreads * i) >> 2));
    philox4x32_10_folded((uint32_t)m, (uint32_t)(m >> 32), a.fk, w[i]);
    philox4x32_10_folded((uint32_t)m, (uint32_t)(m >> 32), a.fk_b, w[G + i]);
  }
  unsigned long long x2[2 * G][2], r2[2 * G][2];
  normal_parts_groups_x2_packed<2 * G>(w, a.coeffs.central2, a.coeffs.tail, x2, r2);
#pragma unroll
  for (int i = 0; i < G; ++i) {
    const uint32_t o = off + 4u * kThreads * i;
    if (o >= len) continue;
    float v[4][4];
#pragma unroll
    for (int s = 0; s < 2; ++s)
#pragma unroll
      for (int p = 0; p < 2; ++p) {
        const unsigned long long t2 = pack_f32x2(th[i][2 * p], th[i][2 * p + 1]);
        const unsigned long long xs = x2[s * G + i][p], rs = r2[s * G + i][p];
        unpack_f32x2(fma_f32x2(rs, xs, t2), v[2 * s][2 * p], v[2 * s][2 * p + 1]);
        unpack_f32x2(fma_f32x2(rs, mul_f32x2(xs, splat_f32x2(-1.0f)), t2), v[2 * s + 1][2 * p],
                     v[2 * s + 1][2 * p + 1]);
      }
    store_two_pairs_full<WT>(a, b + o, v);
  }
}

// The two-pairs perturb over an aligned tile whose counters are all below 2^32, in spans of
// kTwoPairsSpan elements.  A full span runs with its length as a compile-time constant and a
// last partial span with a compile-time loop bound and a runtime exit: with the tile length
// as the loop bound the step spilled 72 bytes a thread and the launch took 1.11 ms per
// 503M-element subspace, against 1.03 ms for these forms.
constexpr uint32_t kTwoPairsSpan = 16384;

template <typename WT, int G, bool FULL>
__device__ __forceinline__ void two_pairs_span(const ElemArgs &a, uint64_t b, uint32_t n) {
  const float *__restrict__ mt = a.master + b;
  const uint32_t q0_lo = (uint32_t)(b >> 2);
  const uint32_t len = FULL ? kTwoPairsSpan : n;
  for (uint32_t off = 4u * threadIdx.x; off < kTwoPairsSpan; off += 4u * kThreads * G) {
    if (!FULL && off >= len) break;
    float th[G][4];
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint32_t o = off + 4u * kThreads * i;
      if (FULL || o < len) {
        const float4 v = ld_stream_f4(mt + o);
        th[i][0] = v.x, th[i][1] = v.y, th[i][2] = v.z, th[i][3] = v.w;
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) th[i][k] = 0.0f;
      }
    }
    two_pairs_step<WT, G>(a, b, len, off, q0_lo, th);
  }
}

template <typename WT, int G>
__device__ __forceinline__ void two_pairs_tile(const ElemArgs &a, uint64_t b, uint32_t len) {
  static_assert(kTwoPairsSpan % (4 * kThreads * G) == 0, "a full span is whole steps");
  uint32_t c0 = 0;
  for (; len - c0 >= kTwoPairsSpan; c0 += kTwoPairsSpan) two_pairs_span<WT, G, true>(a, b + c0, kTwoPairsSpan);
  if (c0 < len) two_pairs_span<WT, G, false>(a, b + c0, len - c0);
}

// Tile whose ends are multiples of 4: every group is whole.  Tile-local pointers and
// 32-bit offsets; G groups per thread per step, loads issued before the math.
// HI0: every counter of the tile is below 2^32 (its high word is the constant 0), so the
// counter arithmetic stays in 32 bits and the compiler drops Philox's first-round
// multiply of word 2 and hoists the second round's multiply of word 0; the pair perturb
// then takes the G groups together (pair_perturb_step).
template <int OP, typename WT, int G, bool HI0>
__device__ __forceinline__ void elem_tile_aligned(const ElemArgs &a, uint64_t b, uint32_t len) {
  float *__restrict__ mt = a.master + b;
  const uint64_t q0 = b >> 2;
  const uint32_t q0_lo = (uint32_t)q0;
  for (uint32_t off = 4u * threadIdx.x; off < len; off += 4u * kThreads * G) {
    float th[G][4];
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint32_t o = off + 4u * kThreads * i;
      if (OP != kOpInit && o < len) {
        const float4 v = ld_stream_f4(mt + o);
        th[i][0] = v.x, th[i][1] = v.y, th[i][2] = v.z, th[i][3] = v.w;
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) th[i][k] = 0.0f;
      }
    }
    if constexpr (OP == kOpPerturbPair && HI0) {
      pair_perturb_step<WT, G>(a, b, len, off, q0_lo, th);
      continue;
    }
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint32_t o = off + 4u * kThreads * i;
      if (o >= len) continue;
      if constexpr (OP == kOpPerturbTwoPairs) {
        const uint64_t q = q0 + (o >> 2);
        float v4[4][4];
        two_pairs_values(a, (uint32_t)q, (uint32_t)(q >> 32), th[i], v4);
        store_two_pairs_full<WT>(a, b + o, v4);
        continue;
      }
      float v[4], vp[4];
      if (HI0) {
        elem_values<OP>(a, q0_lo + (o >> 2), 0u, th[i], v, vp);
      } else {
        const uint64_t q = q0 + (o >> 2);
        elem_values<OP>(a, (uint32_t)q, (uint32_t)(q >> 32), th[i], v, vp);
      }
      if (OP == kOpInit) st_stream_f4(mt + o, make_float4(v[0], v[1], v[2], v[3]));
      WStore<WT>::full(a.w, b + o, v);
      if (writes_context<OP>()) store_copies_full<WT>(a.copies, b + o, v);
      if (OP == kOpPerturbPair) WStore<WT>::full(a.partner, b + o - a.partner_base, vp);
    }
  }
}

// General tile: groups cut by the tile's ends are handled element by element.
template <int OP, typename WT, int G>
__device__ __forceinline__ void elem_tile_ragged(const ElemArgs &a, uint64_t b, uint64_t e) {
  float *__restrict__ master = a.master;
  const uint64_t lo = b & ~3ull;
  for (uint64_t base = lo + 4ull * threadIdx.x; base < e; base += 4ull * kThreads * G) {
    float th[G][4];
    bool full[G];
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint64_t g4 = base + 4ull * kThreads * i;
      full[i] = g4 >= b && g4 + 4 <= e;
      if (OP != kOpInit) {
        if (full[i]) {
          const float4 v = ld_stream_f4(master + g4);
          th[i][0] = v.x, th[i][1] = v.y, th[i][2] = v.z, th[i][3] = v.w;
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k)
            th[i][k] = (g4 + k >= b && g4 + k < e) ? master[g4 + k] : 0.0f;
        }
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) th[i][k] = 0.0f;
      }
    }
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint64_t g4 = base + 4ull * kThreads * i;
      if (g4 >= e) continue;
      if constexpr (OP == kOpPerturbTwoPairs) {
        float v4[4][4];
        two_pairs_values(a, (uint32_t)(g4 >> 2), (uint32_t)(g4 >> 34), th[i], v4);
        if (full[i]) {
          store_two_pairs_full<WT>(a, g4, v4);
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (g4 + k >= b && g4 + k < e) store_two_pairs_one<WT>(a, g4 + k, v4, k);
        }
        continue;
      }
      float v[4], vp[4];
      elem_values<OP>(a, (uint32_t)(g4 >> 2), (uint32_t)(g4 >> 34), th[i], v, vp);
      if (full[i]) {
        if (OP == kOpInit) st_stream_f4(master + g4, make_float4(v[0], v[1], v[2], v[3]));
        WStore<WT>::full(a.w, g4, v);
        if (writes_context<OP>()) store_copies_full<WT>(a.copies, g4, v);
        if (OP == kOpPerturbPair) WStore<WT>::full(a.partner, g4 - a.partner_base, vp);
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint64_t g = g4 + k;
          if (g >= b && g < e) {
            if (OP == kOpInit) master[g] = v[k];
            WStore<WT>::one(a.w, g, v[k]);
            if (writes_context<OP>()) store_copies_one<WT>(a.copies, g, v[k]);
            if (OP == kOpPerturbPair) WStore<WT>::one(a.partner, g - a.partner_base, vp[k]);
          }
        }
      }
    }
  }
}

// One block per tile [tiles[2t], tiles[2t+1]).  Launch shapes, measured on the 4B set:
// the pair perturb takes G = 4 groups per step together (one tail vote for the four) at 4
// resident blocks per SM (64 registers a thread): 0.603 ms against 0.631 ms for G = 8 one
// group at a time at 3 blocks.  The two-pairs perturb takes G = 1 group (2 Philox blocks
// per step, packed steps) at 4 blocks per SM (56 registers, no spill): 1.054 ms per
// 503M-element subspace, against 1.088 ms at 5 blocks and, in an earlier form, 1.1-2.3%
// more for G = 2 (scalar steps, or packed with 52 bytes a thread spilled).  The other ops
// take G = 8 groups one at a time at 3 blocks per SM (85 registers), which the plain
// perturb runs faster (0.532 against 0.544 ms).
template <int OP>
constexpr int elem_blocks_per_sm() { return OP == kOpPerturbPair || OP == kOpPerturbTwoPairs ? 4 : 3; }
template <int OP>
constexpr int elem_groups() { return OP == kOpPerturbPair ? 4 : (OP == kOpPerturbTwoPairs ? 1 : 8); }

// A tile outside [partner_base, partner_base + partner_len) is skipped and flagged.
__device__ __forceinline__ bool partner_covers(const ElemArgs &a, uint64_t b, uint64_t e) {
  return b >= a.partner_base && e - a.partner_base <= a.partner_len;
}

template <int OP, typename WT, int G>
__global__ void __launch_bounds__(kThreads, elem_blocks_per_sm<OP>())
    elem_tiles_kernel(const __grid_constant__ ElemArgs a) {
  const uint64_t t = blockIdx.x;
  const uint64_t b = a.tiles[2 * t], e = a.tiles[2 * t + 1];
  if (b > e || e > a.n_alloc || e - b > (uint64_t)COPES_TILE_MAX) {
    if (threadIdx.x == 0) flag_error(kErrTileRange);
    return;
  }
  if (OP == kOpPerturbPair && !partner_covers(a, b, e)) {
    if (threadIdx.x == 0) flag_error(kErrPartnerRange);
    return;
  }
  if constexpr (OP == kOpPerturbTwoPairs) {
    // a tile of exactly one span (the default tile size) runs the span with every bound
    // a compile-time constant: 1.054 ms per 503M-element subspace against 1.110 ms through
    // the span loop of two_pairs_tile
    if (((b | e) & 3ull) == 0 && (e >> 34) == 0) {
      if (e - b == kTwoPairsSpan) two_pairs_span<WT, G, true>(a, b, kTwoPairsSpan);
      else two_pairs_tile<WT, G>(a, b, (uint32_t)(e - b));
    } else if (((b | e) & 3ull) == 0) {
      elem_tile_aligned<OP, WT, G, false>(a, b, (uint32_t)(e - b));
    } else {
      elem_tile_ragged<OP, WT, G>(a, b, e);
    }
    return;
  }
  if (((b | e) & 3ull) == 0) {
    if ((e >> 34) == 0) elem_tile_aligned<OP, WT, G, true>(a, b, (uint32_t)(e - b));
    else elem_tile_aligned<OP, WT, G, false>(a, b, (uint32_t)(e - b));
  } else {
    elem_tile_ragged<OP, WT, G>(a, b, e);
  }
}

// The partner member's perturb over TILES: w[g] = partner[g - partner_base], a copy of
// the working dtype's bits (the values kOpPerturbPair wrote).  Aligned tiles move one
// 4-element group (8 B bf16, 16 B fp32) per load; ragged tiles go element by element.
template <typename WT>
struct Group4;
template <>
struct Group4<__nv_bfloat16> {
  using T = uint2;
};
template <>
struct Group4<float> {
  using T = uint4;
};

template <typename WT, int G>
__global__ void __launch_bounds__(kThreads) partner_tiles_kernel(const ElemArgs a) {
  const uint64_t t = blockIdx.x;
  const uint64_t b = a.tiles[2 * t], e = a.tiles[2 * t + 1];
  if (b > e || e > a.n_alloc || e - b > (uint64_t)COPES_TILE_MAX) {
    if (threadIdx.x == 0) flag_error(kErrTileRange);
    return;
  }
  if (!partner_covers(a, b, e)) {
    if (threadIdx.x == 0) flag_error(kErrPartnerRange);
    return;
  }
  const WT *__restrict__ src = reinterpret_cast<const WT *>(a.partner) + (b - a.partner_base);
  WT *__restrict__ dst = reinterpret_cast<WT *>(a.w) + b;
  const uint32_t len = (uint32_t)(e - b);
  if (((b | e) & 3ull) == 0) {  // partner_base is a multiple of 4, so src is aligned too
    using V = typename Group4<WT>::T;
    const V *__restrict__ vs = reinterpret_cast<const V *>(src);
    V *__restrict__ vd = reinterpret_cast<V *>(dst);
    const uint32_t n = len / 4;
    for (uint32_t i0 = threadIdx.x; i0 < n; i0 += kThreads * G) {
      V v[G];
#pragma unroll
      for (int k = 0; k < G; ++k)
        if (i0 + kThreads * k < n) v[k] = __ldcs(vs + i0 + kThreads * k);
#pragma unroll
      for (int k = 0; k < G; ++k)
        if (i0 + kThreads * k < n) __stcs(vd + i0 + kThreads * k, v[k]);
    }
  } else {
    for (uint32_t i = threadIdx.x; i < len; i += kThreads) dst[i] = src[i];
  }
}

// Gather form: the block's segment of the sorted index list is staged into shared memory
// chunk by chunk (TMA bulk copies, double-buffered); each thread then handles its indices
// of the chunk: load theta[g], one Philox word's normal, store w[g] (and theta[g] for init).
// GATH: theta lives in the subspace's gathered copy at the index's list position p
// (a.gathered[p]) instead of master[g]; kOpGather / kOpScatter copy between the two.
template <int OP, typename WT, bool GATH>
__global__ void __launch_bounds__(kThreads) elem_index_kernel(const ElemArgs a) {
  __shared__ __align__(128) int64_t s_idx[2][kStageChunk];
  __shared__ __align__(8) uint64_t s_bar[2];
  constexpr int U = kStageChunk / kThreads;
  const uint64_t s0 = (uint64_t)blockIdx.x * kIndexSegment;
  const uint64_t s1 = min(s0 + (uint64_t)kIndexSegment, a.n_index);
  float *__restrict__ master = a.master;
  float *__restrict__ gath = a.gathered;
  staged_index_segment(a.index, s0, s1, s_idx, s_bar, [] { flag_error(kErrStageTimeout); },
                       [&](const int64_t *chunk, int cnt, uint64_t first) {
    int64_t g[U];
    float th[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int p = threadIdx.x + kThreads * u;
      ok[u] = p < cnt;
      g[u] = ok[u] ? chunk[p] : 0;
      if (ok[u] && (g[u] < 0 || (uint64_t)g[u] >= a.n_alloc)) {
        flag_error(kErrIndexRange);
        ok[u] = false;
      }
      if ((OP == kOpPerturbPair || OP == kOpPartner) && ok[u] &&
          ((uint64_t)g[u] < a.partner_base || (uint64_t)g[u] - a.partner_base >= a.partner_len)) {
        flag_error(kErrPartnerRange);
        ok[u] = false;
      }
      const bool from_gathered = GATH && OP != kOpGather;
      const bool reads_theta = OP != kOpInit && OP != kOpPartner;
      th[u] = (reads_theta && ok[u]) ? (from_gathered ? gath[first + p] : master[g[u]]) : 0.0f;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      if constexpr (OP == kOpGather) {
        gath[first + threadIdx.x + kThreads * u] = th[u];
        continue;
      } else if constexpr (OP == kOpScatter) {
        master[g[u]] = th[u];
        continue;
      } else if constexpr (OP == kOpPartner) {
        const uint64_t gi = (uint64_t)g[u];
        reinterpret_cast<WT *>(a.w)[gi] = reinterpret_cast<const WT *>(a.partner)[gi - a.partner_base];
        continue;
      } else {
        float v, vp = 0.0f;
        if (OP == kOpRestore) {
          v = th[u];
        } else {
          uint32_t x[4];
          const uint64_t q = (uint64_t)g[u] >> 2;
          philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, op_tag<OP>(), a.rk, x);
          const uint32_t sel = (uint32_t)g[u] & 3u;
          const uint32_t wd = sel == 0 ? x[0] : (sel == 1 ? x[1] : (sel == 2 ? x[2] : x[3]));
          float xv, r;
          normal_parts(wd, a.coeffs.central, a.coeffs.tail, xv, r);  // r = a * R(L)
          v = __fmaf_rn(r, xv, OP == kOpInit ? a.b : th[u]);
          if (OP == kOpPerturbPair) vp = __fmaf_rn(-r, xv, th[u]);
        }
        if (OP == kOpInit) {
          if (GATH) gath[first + threadIdx.x + kThreads * u] = v;
          else master[g[u]] = v;
        }
        WStore<WT>::one(a.w, (uint64_t)g[u], v);
        if (writes_context<OP>()) store_copies_one<WT>(a.copies, (uint64_t)g[u], v);
        if (OP == kOpPerturbPair) WStore<WT>::one(a.partner, (uint64_t)g[u] - a.partner_base, vp);
      }
    }
  });
}

template <int OP, typename WT>
static cudaError_t launch_elem_typed(int kind, const ElemArgs &a, cudaStream_t s) {
  if constexpr (OP == kOpPerturbTwoPairs) {
    if (kind != COPES_SUBSPACE_TILES || a.copies.n != 3) return cudaErrorInvalidValue;
    if (a.n_tiles == 0) return cudaSuccess;
    elem_tiles_kernel<OP, WT, elem_groups<OP>()><<<(unsigned)a.n_tiles, kThreads, 0, s>>>(a);
  } else if constexpr (OP == kOpGather || OP == kOpScatter) {
    if (kind != COPES_SUBSPACE_INDICES || !a.gathered) return cudaErrorInvalidValue;
    if (a.n_index == 0) return cudaSuccess;
    const uint64_t blocks = (a.n_index + kIndexSegment - 1) / kIndexSegment;
    elem_index_kernel<OP, WT, true><<<(unsigned)blocks, kThreads, 0, s>>>(a);
  } else if (kind == COPES_SUBSPACE_TILES) {
    if (a.n_tiles == 0) return cudaSuccess;
    constexpr int G = elem_groups<OP>();
    if constexpr (OP == kOpPartner)
      partner_tiles_kernel<WT, G><<<(unsigned)a.n_tiles, kThreads, 0, s>>>(a);
    else
      elem_tiles_kernel<OP, WT, G><<<(unsigned)a.n_tiles, kThreads, 0, s>>>(a);
  } else {
    if (a.n_index == 0) return cudaSuccess;
    const uint64_t blocks = (a.n_index + kIndexSegment - 1) / kIndexSegment;
    if (a.gathered) elem_index_kernel<OP, WT, true><<<(unsigned)blocks, kThreads, 0, s>>>(a);
    else elem_index_kernel<OP, WT, false><<<(unsigned)blocks, kThreads, 0, s>>>(a);
  }
  return cudaGetLastError();
}

template <int OP>
static cudaError_t launch_elem_op(int kind, int dtype, const ElemArgs &a, cudaStream_t s) {
  return dtype == COPES_BF16 ? launch_elem_typed<OP, __nv_bfloat16>(kind, a, s)
                             : launch_elem_typed<OP, float>(kind, a, s);
}

cudaError_t launch_elementwise(int op, int kind, int dtype, const ElemArgs &a, cudaStream_t s) {
  switch (op) {
    case kOpPerturb: return launch_elem_op<kOpPerturb>(kind, dtype, a, s);
    case kOpRestore: return launch_elem_op<kOpRestore>(kind, dtype, a, s);
    case kOpGather: return launch_elem_op<kOpGather>(kind, dtype, a, s);
    case kOpScatter: return launch_elem_op<kOpScatter>(kind, dtype, a, s);
    case kOpPerturbPair: return launch_elem_op<kOpPerturbPair>(kind, dtype, a, s);
    case kOpPartner: return launch_elem_op<kOpPartner>(kind, dtype, a, s);
    case kOpPerturbTwoPairs: return launch_elem_op<kOpPerturbTwoPairs>(kind, dtype, a, s);
    default: return launch_elem_op<kOpInit>(kind, dtype, a, s);
  }
}

// ------------------------------------------------------------------------- update
// One block per tile: the prologue (noise_weights_to_smem) folds the members into one
// weight per noise vector; every thread then regenerates all P noise vectors for its G
// groups in registers (noise_sum_groups), acc = sum_j w_j eps_j (j ascending), and
// writes theta = fma(coef, acc, theta) and, with COMMIT, its rounding to the working
// copies.
template <typename WT, int G, bool COMMIT, bool HI0>
__device__ __forceinline__ void update_tile(const UpdateArgs &a, const float *s_w,
                                            const uint32_t (*s_rk)[20], const uint32_t (*s_fk)[20],
                                            uint64_t b, uint64_t e) {
  float *__restrict__ master = a.master;
  const uint64_t lo = b & ~3ull;
  for (uint64_t base = lo + 4ull * threadIdx.x; base < e; base += 4ull * kThreads * G) {
    float acc[G][4];
    noise_sum_groups<G, HI0>(base, a.n_noise, s_w, s_rk, s_fk, acc);
    // theta is read only now, after the noise loop, so it occupies no registers there
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint64_t g4 = base + 4ull * kThreads * i;
      if (g4 >= e) continue;
      if (g4 >= b && g4 + 4 <= e) {
        const float4 t = ld_stream_f4(master + g4);
        float v[4] = {__fmaf_rn(a.coef, acc[i][0], t.x), __fmaf_rn(a.coef, acc[i][1], t.y),
                      __fmaf_rn(a.coef, acc[i][2], t.z), __fmaf_rn(a.coef, acc[i][3], t.w)};
        st_stream_f4(master + g4, make_float4(v[0], v[1], v[2], v[3]));
        if (COMMIT) {
          WStore<WT>::full(a.w, g4, v);
          store_copies_full<WT>(a.copies, g4, v);
        }
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint64_t g = g4 + k;
          if (g >= b && g < e) {
            const float v = __fmaf_rn(a.coef, acc[i][k], master[g]);
            master[g] = v;
            if (COMMIT) {
              WStore<WT>::one(a.w, g, v);
              store_copies_one<WT>(a.copies, g, v);
            }
          }
        }
      }
    }
  }
}

// update_tile for an aligned tile of exactly kUpdateSpan elements (the default tile size)
// whose counters are below 2^32, with the tile loop's bounds compile-time constants and
// no edge tests: 7.455 against 7.568 ms per 503M-element subspace at P = 16, the same
// values bit for bit.
constexpr uint32_t kUpdateSpan = 16384;

template <typename WT, int G, bool COMMIT>
__device__ __forceinline__ void update_tile_full(const UpdateArgs &a, const float *s_w,
                                                 const uint32_t (*s_rk)[20], const uint32_t (*s_fk)[20],
                                                 uint64_t b) {
  static_assert(kUpdateSpan % (4 * kThreads * G) == 0, "a full tile is whole steps");
  float *__restrict__ mt = a.master + b;
  for (uint32_t off = 4u * threadIdx.x; off < kUpdateSpan; off += 4u * kThreads * G) {
    float acc[G][4];
    noise_sum_groups<G, true>(b + off, a.n_noise, s_w, s_rk, s_fk, acc);
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint32_t o = off + 4u * kThreads * i;
      const float4 t = ld_stream_f4(mt + o);
      float v[4] = {__fmaf_rn(a.coef, acc[i][0], t.x), __fmaf_rn(a.coef, acc[i][1], t.y),
                    __fmaf_rn(a.coef, acc[i][2], t.z), __fmaf_rn(a.coef, acc[i][3], t.w)};
      st_stream_f4(mt + o, make_float4(v[0], v[1], v[2], v[3]));
      if (COMMIT) {
        WStore<WT>::full(a.w, b + o, v);
        store_copies_full<WT>(a.copies, b + o, v);
      }
    }
  }
}

// Launch shape of the tile update: groups per thread and resident blocks per SM
// (registers: 65536 / (256 x blocks) a thread).  Measured best for P = 4, 16 and 64.
constexpr int kUpdateGroups = 2;
constexpr int kUpdateBlocksPerSM = 4;

// One block per tile; the prologue folds the members into noise weights and expands each
// noise vector's Philox keys (round keys, and the folded form) into shared memory.
template <typename WT, int G, bool COMMIT, int BLOCKS>
__global__ void __launch_bounds__(kThreads, BLOCKS) update_tiles_kernel(const __grid_constant__ UpdateArgs a) {
  __shared__ float s_w[COPES_MAX_NOISE];
  __shared__ __align__(16) uint32_t s_rk[COPES_MAX_NOISE][20];
  __shared__ __align__(16) uint32_t s_fk[COPES_MAX_NOISE][20];
  noise_weights_to_smem(a, s_w, s_rk, s_fk);
  const uint64_t t = blockIdx.x;
  const uint64_t b = a.tiles[2 * t], e = a.tiles[2 * t + 1];
  if (b > e || e > a.n_alloc || e - b > (uint64_t)COPES_TILE_MAX) {
    if (threadIdx.x == 0) flag_error(kErrTileRange);
    return;
  }
  if (e - b == kUpdateSpan && (b & 3ull) == 0 && (e >> 34) == 0) update_tile_full<WT, G, COMMIT>(a, s_w, s_rk, s_fk, b);
  else if ((e >> 34) == 0) update_tile<WT, G, COMMIT, true>(a, s_w, s_rk, s_fk, b, e);
  else update_tile<WT, G, COMMIT, false>(a, s_w, s_rk, s_fk, b, e);
}

// Gather form of the update: indices staged through shared memory as in
// elem_index_kernel; every index regenerates the P normals from its own Philox word.
// GATH: theta is read from and written to the gathered copy at the list position.
template <typename WT, bool COMMIT, bool GATH>
__global__ void __launch_bounds__(kThreads) update_index_kernel(const __grid_constant__ UpdateArgs a) {
  __shared__ float s_w[COPES_MAX_NOISE];
  __shared__ __align__(16) uint32_t s_rk[COPES_MAX_NOISE][20];
  __shared__ __align__(128) int64_t s_idx[2][kStageChunk];
  __shared__ __align__(8) uint64_t s_bar[2];
  noise_weights_to_smem(a, s_w, s_rk);
  constexpr int U = 2;
  const uint64_t s0 = (uint64_t)blockIdx.x * kIndexSegment;
  const uint64_t s1 = min(s0 + (uint64_t)kIndexSegment, a.n_index);
  float *__restrict__ master = a.master;
  float *__restrict__ gath = a.gathered;
  const int P = a.n_noise;
  staged_index_segment(a.index, s0, s1, s_idx, s_bar, [] { flag_error(kErrStageTimeout); },
                       [&](const int64_t *chunk, int cnt, uint64_t first) {
    for (int p0 = threadIdx.x; p0 < cnt; p0 += kThreads * U) {
      int64_t g[U];
      float acc[U];
      bool ok[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int p = p0 + kThreads * u;
        ok[u] = p < cnt;
        g[u] = ok[u] ? chunk[p] : 0;
        if (ok[u] && (g[u] < 0 || (uint64_t)g[u] >= a.n_alloc)) {
          flag_error(kErrIndexRange);
          ok[u] = false;
        }
        acc[u] = 0.0f;
      }
      for (int j = 0; j < P; ++j) {
        uint32_t rk[20];
#pragma unroll
        for (int r = 0; r < 20; r += 4) {
          const uint4 v = *reinterpret_cast<const uint4 *>(&s_rk[j][r]);
          rk[r] = v.x, rk[r + 1] = v.y, rk[r + 2] = v.z, rk[r + 3] = v.w;
        }
        const float wj = s_w[j];
        uint32_t wd[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          uint32_t x[4];
          const uint64_t q = (uint64_t)g[u] >> 2;
          philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, COPES_TAG_NOISE, rk, x);
          const uint32_t sel = (uint32_t)g[u] & 3u;
          wd[u] = sel == 0 ? x[0] : (sel == 1 ? x[1] : (sel == 2 ? x[2] : x[3]));
        }
        // the two indices' normals as one packed pair (bit-identical to one at a time)
        static_assert(U == 2, "normals are paired");
        float eps0, eps1;
        normal_pair_x2(wd[0], wd[1], eps0, eps1);
        acc[0] = __fmaf_rn(wj, eps0, acc[0]);
        acc[1] = __fmaf_rn(wj, eps1, acc[1]);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (!ok[u]) continue;
        float *th = GATH ? &gath[first + p0 + kThreads * u] : &master[g[u]];
        const float v = __fmaf_rn(a.coef, acc[u], *th);
        *th = v;
        if (COMMIT) {
          WStore<WT>::one(a.w, (uint64_t)g[u], v);
          store_copies_one<WT>(a.copies, (uint64_t)g[u], v);
        }
      }
    }
  });
}

template <typename WT, bool COMMIT>
static cudaError_t launch_update_typed(int kind, const UpdateArgs &a, cudaStream_t s) {
  if (kind == COPES_SUBSPACE_TILES) {
    if (a.n_tiles == 0) return cudaSuccess;
    update_tiles_kernel<WT, kUpdateGroups, COMMIT, kUpdateBlocksPerSM><<<(unsigned)a.n_tiles, kThreads, 0, s>>>(a);
  } else {
    if (a.n_index == 0) return cudaSuccess;
    const uint64_t blocks = (a.n_index + kIndexSegment - 1) / kIndexSegment;
    if (a.gathered) update_index_kernel<WT, COMMIT, true><<<(unsigned)blocks, kThreads, 0, s>>>(a);
    else update_index_kernel<WT, COMMIT, false><<<(unsigned)blocks, kThreads, 0, s>>>(a);
  }
  return cudaGetLastError();
}

cudaError_t launch_update(int kind, int dtype, const UpdateArgs &a, cudaStream_t s, int) {
  if (dtype == COPES_BF16)
    return a.fuse_commit ? launch_update_typed<__nv_bfloat16, true>(kind, a, s)
                         : launch_update_typed<__nv_bfloat16, false>(kind, a, s);
  return a.fuse_commit ? launch_update_typed<float, true>(kind, a, s)
                       : launch_update_typed<float, false>(kind, a, s);
}

// -------------------------------------------------------------------------- debug
__global__ void debug_philox_kernel(uint64_t seed, uint64_t q0, uint64_t n, uint32_t aux,
                                    uint32_t tag, uint32_t *out) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint64_t q = q0 + i;
  uint32_t rk[20], x[4];
  philox_round_keys((uint32_t)seed, (uint32_t)(seed >> 32), rk);
  philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), aux, tag, rk, x);
  reinterpret_cast<uint4 *>(out)[i] = make_uint4(x[0], x[1], x[2], x[3]);
}

__global__ void debug_normals_kernel(uint64_t seed, uint32_t tag, uint64_t g0, uint64_t n,
                                     float *out) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  out[i] = index_noise(g0 + i, tag, (uint32_t)seed, (uint32_t)(seed >> 32));
}

__global__ void debug_transform_kernel(const uint32_t *words, uint64_t n, float *out) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = normal_from_word(words[i]);
}

static unsigned blocks_for(uint64_t n) { return (unsigned)((n + kThreads - 1) / kThreads); }

cudaError_t launch_debug_philox(uint64_t seed, uint64_t q0, uint64_t n, uint32_t aux,
                                uint32_t tag, uint32_t *out, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  debug_philox_kernel<<<blocks_for(n), kThreads, 0, s>>>(seed, q0, n, aux, tag, out);
  return cudaGetLastError();
}

cudaError_t launch_debug_normals(uint64_t seed, uint32_t tag, uint64_t g0, uint64_t n,
                                 float *out, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  debug_normals_kernel<<<blocks_for(n), kThreads, 0, s>>>(seed, tag, g0, n, out);
  return cudaGetLastError();
}

cudaError_t launch_debug_transform(const uint32_t *words, uint64_t n, float *out,
                                   cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  debug_transform_kernel<<<blocks_for(n), kThreads, 0, s>>>(words, n, out);
  return cudaGetLastError();
}

unsigned read_and_clear_es_errors() {
  unsigned v = 0, zero = 0;
  cudaMemcpyFromSymbol(&v, g_es_error, sizeof(v));
  if (v) cudaMemcpyToSymbol(g_es_error, &zero, sizeof(zero));
  return v;
}

}  // namespace copes
