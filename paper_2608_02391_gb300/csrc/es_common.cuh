// Device pieces shared by the ES kernels of the tile / gather path (es_kernels.cu) and of
// the partition-replay path (replay_kernels.cu): working-weight stores and the update's
// prologue.
#pragma once

#include <cuda_bf16.h>

#include "copes_device.cuh"
#include "copes_internal.h"

namespace copes {

template <typename WT>
struct WStore;

template <>
struct WStore<__nv_bfloat16> {
  static __device__ __forceinline__ void full(void *w, uint64_t g, const float v[4]) {
    uint2 p;
    p.x = pack_bf16x2(v[0], v[1]);
    p.y = pack_bf16x2(v[2], v[3]);
    st_stream_u2(reinterpret_cast<uint16_t *>(w) + g, p);
  }
  static __device__ __forceinline__ void one(void *w, uint64_t g, float v) {
    reinterpret_cast<uint16_t *>(w)[g] = to_bf16_bits(v);
  }
};

template <>
struct WStore<float> {
  static __device__ __forceinline__ void full(void *w, uint64_t g, const float v[4]) {
    st_stream_f4(reinterpret_cast<float *>(w) + g, make_float4(v[0], v[1], v[2], v[3]));
  }
  static __device__ __forceinline__ void one(void *w, uint64_t g, float v) {
    reinterpret_cast<float *>(w)[g] = v;
  }
};

// The context's stores to the working copies beyond w (restore / commit / init and the
// update's fused commit).
template <typename WT>
__device__ __forceinline__ void store_copies_full(const WorkingCopies &c, uint64_t g, const float v[4]) {
#pragma unroll
  for (int i = 0; i < 3; ++i)
    if (i < c.n) WStore<WT>::full(c.p[i], g, v);
}

template <typename WT>
__device__ __forceinline__ void store_copies_one(const WorkingCopies &c, uint64_t g, float v) {
#pragma unroll
  for (int i = 0; i < 3; ++i)
    if (i < c.n) WStore<WT>::one(c.p[i], g, v);
}

// The update's prologue: folds the members into one weight per noise vector,
//   w_j = sum_{i : noise(i) = j} sign_i f_i  (member order, fp32),
// and expands each noise vector's Philox round keys into shared memory (and, when s_fk is
// given, the folded keys of philox4x32_10_folded for the noise tag).
__device__ __forceinline__ void noise_weights_to_smem(const UpdateArgs &a, float *s_w,
                                                      uint32_t (*s_rk)[20],
                                                      uint32_t (*s_fk)[20] = nullptr) {
  for (int j = threadIdx.x; j < a.n_noise; j += blockDim.x) {
    philox_round_keys(a.seed_lo[j], a.seed_hi[j], s_rk[j]);
    if (s_fk) philox_folded_keys(s_rk[j], COPES_TAG_NOISE, s_fk[j]);
    float acc = 0.0f;
    for (int m = a.noise_ptr[j]; m < a.noise_ptr[j + 1]; ++m) {
      const int i = a.noise_member[m];
      const float f = a.fitness[i];
      acc = __fadd_rn(acc, a.sign[i] > 0 ? f : -f);
    }
    s_w[j] = acc;
  }
  __syncthreads();
}

// The update's noise sum for the G groups of one thread, the 4-element groups at
// base + 4 kThreads i: acc[i][k] = sum_j w_j eps_j[g] over the P noise vectors, j
// ascending, each term one fp32 fma.  Per noise vector the G groups' Philox calls run
// first, then their transforms with one tail vote (normal_parts_groups_packed), then the
// accumulation; the transform and the accumulation run on packed fp32 pairs (the values
// of scalar steps, bit for bit).  HI0 (every counter below 2^32): Philox in the folded
// form (s_fk), with each group's product M0 * q computed once for all noise vectors;
// otherwise the plain form with 64-bit counters (s_rk).
template <int G, bool HI0>
__device__ __forceinline__ void noise_sum_groups(uint64_t base, int P, const float *s_w,
                                                 const uint32_t (*s_rk)[20], const uint32_t (*s_fk)[20],
                                                 float (&acc)[G][4]) {
  unsigned long long acc2[G][2];  // the accumulators of group i as pairs (2p, 2p + 1)
#pragma unroll
  for (int i = 0; i < G; ++i) acc2[i][0] = acc2[i][1] = 0ull;
  const uint32_t q_lo = (uint32_t)(base >> 2);  // counter of group 0 (HI0: the whole counter)
  uint32_t m0_lo[G], m0_hi[G];                  // HI0: M0 * counter of each group
  if (HI0) {
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint64_t m = (uint64_t)kPhiloxM0 * (q_lo + kThreads * i);
      m0_lo[i] = (uint32_t)m;
      m0_hi[i] = (uint32_t)(m >> 32);
    }
  }
  for (int j = 0; j < P; ++j) {
    uint32_t k[20];
    const uint32_t *src = HI0 ? s_fk[j] : s_rk[j];
#pragma unroll
    for (int r = 0; r < 20; r += 4) {
      const uint4 v = *reinterpret_cast<const uint4 *>(src + r);
      k[r] = v.x, k[r + 1] = v.y, k[r + 2] = v.z, k[r + 3] = v.w;
    }
    const float wj = s_w[j];
    uint32_t w[G][4];
#pragma unroll
    for (int i = 0; i < G; ++i) {
      if (HI0) {
        philox4x32_10_folded(m0_lo[i], m0_hi[i], k, w[i]);
      } else {
        const uint64_t q = (base >> 2) + kThreads * i;
        philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, COPES_TAG_NOISE, k, w[i]);
      }
    }
    unsigned long long x2[G][2], r2[G][2];
    normal_parts_groups_packed<G>(w, x2, r2);
#pragma unroll
    for (int i = 0; i < G; ++i)
#pragma unroll
      for (int p = 0; p < 2; ++p) acc2[i][p] = fma_f32x2(splat_f32x2(wj), mul_f32x2(x2[i][p], r2[i][p]), acc2[i][p]);
  }
#pragma unroll
  for (int i = 0; i < G; ++i) {
    unpack_f32x2(acc2[i][0], acc[i][0], acc[i][1]);
    unpack_f32x2(acc2[i][1], acc[i][2], acc[i][3]);
  }
}

}  // namespace copes
