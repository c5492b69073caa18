// Fitness shaping of the population's rewards: population z-score (Eq. 5 / Eq. 12),
// per-group z-score (the independent standardisation of Sec. 4.4), centred ranks, or
// identity.  One block of COPES_MAX_MEMBERS threads; statistics in fp64 with
// warp-shuffle reductions.
#include <math.h>

#include "copes_internal.h"

namespace copes {

constexpr int kShapeThreads = COPES_MAX_MEMBERS;
constexpr int kShapeWarps = kShapeThreads / 32;

template <typename T, typename Op>
__device__ __forceinline__ T block_reduce(T v, Op op, T *scratch) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, off));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();  // scratch may still be read by a previous reduction
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  T r = scratch[0];
  for (int w = 1; w < kShapeWarps; ++w) r = op(r, scratch[w]);
  return r;
}

struct AddD {
  __device__ double operator()(double a, double b) const { return a + b; }
};
struct MinF {
  __device__ float operator()(float a, float b) const { return fminf(a, b); }
};
struct MaxF {
  __device__ float operator()(float a, float b) const { return fmaxf(a, b); }
};

__global__ void __launch_bounds__(kShapeThreads) shape_kernel(const float *r, int n,
                                                              const int32_t *group, int mode,
                                                              float *f) {
  __shared__ float s_r[kShapeThreads];
  __shared__ int32_t s_g[kShapeThreads];
  __shared__ double s_scratch_d[kShapeWarps];
  __shared__ float s_scratch_f[kShapeWarps];
  const int i = threadIdx.x;
  const bool live = i < n;
  const float ri = live ? r[i] : 0.0f;
  if (live) {
    s_r[i] = ri;
    s_g[i] = (mode == COPES_SHAPE_ZSCORE_GROUPED) ? group[i] : 0;
  }
  __syncthreads();

  if (mode == COPES_SHAPE_NONE) {
    if (live) f[i] = ri;
    return;
  }
  if (mode == COPES_SHAPE_ZSCORE) {
    const double sum = block_reduce(live ? (double)ri : 0.0, AddD(), s_scratch_d);
    const double mean = sum / (double)n;
    const double dev = live ? (double)ri - mean : 0.0;
    const double sq = block_reduce(dev * dev, AddD(), s_scratch_d);
    const float lo = block_reduce(live ? ri : INFINITY, MinF(), s_scratch_f);
    const float hi = block_reduce(live ? ri : -INFINITY, MaxF(), s_scratch_f);
    const double sd = sqrt(sq / (double)n);
    if (live) f[i] = (lo == hi) ? 0.0f : (float)(dev / sd);
    return;
  }
  if (!live) return;
  if (mode == COPES_SHAPE_ZSCORE_GROUPED) {
    const int32_t gi = s_g[i];
    double sum = 0.0;
    int count = 0;
    bool equal = true;
    for (int j = 0; j < n; ++j) {
      if (s_g[j] != gi) continue;
      sum += (double)s_r[j];
      equal = equal && (s_r[j] == ri);
      ++count;
    }
    const double mean = sum / (double)count;
    double sq = 0.0;
    for (int j = 0; j < n; ++j) {
      if (s_g[j] != gi) continue;
      const double d = (double)s_r[j] - mean;
      sq += d * d;
    }
    const double sd = sqrt(sq / (double)count);
    f[i] = equal ? 0.0f : (float)(((double)ri - mean) / sd);
    return;
  }
  // centred ranks: 0-based rank with ties averaged, rank / (n - 1) - 1/2
  if (n == 1) {
    f[i] = 0.0f;
    return;
  }
  int less = 0, equal = 0;
  for (int j = 0; j < n; ++j) {
    less += s_r[j] < ri;
    equal += s_r[j] == ri;
  }
  const double rank = (double)less + 0.5 * (double)(equal - 1);
  f[i] = (float)(rank / (double)(n - 1) - 0.5);
}

cudaError_t launch_shape(const float *r, int n, const int32_t *group, int mode, float *f,
                         cudaStream_t s) {
  shape_kernel<<<1, kShapeThreads, 0, s>>>(r, n, group, mode, f);
  return cudaGetLastError();
}

}  // namespace copes
