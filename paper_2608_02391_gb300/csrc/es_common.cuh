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

}  // namespace copes
