// Partition kernels (Eq. 7; Algorithm 1 "sample a partition"; Supp. A.8 partition
// replay): the hash partition's per-tile histogram, per-bucket exclusive scan and
// order-preserving scatter into sorted int64 lists, and the random-chunk map.
#include "copes_internal.h"

namespace copes {

__device__ unsigned int g_partition_error = 0;

constexpr int kPartThreads = 256;
constexpr int kPartWarps = kPartThreads / 32;

__device__ __forceinline__ uint32_t hash_bucket(uint64_t e, uint32_t tensor_id, uint32_t k0,
                                                uint32_t k1, int K) {
  uint32_t x[4];
  const uint64_t q = e >> 2;
  philox4x32_10((uint32_t)q, (uint32_t)(q >> 32), tensor_id, COPES_TAG_PARTITION, k0, k1, x);
  const uint32_t s = (uint32_t)e & 3u;
  const uint32_t w = s == 0 ? x[0] : (s == 1 ? x[1] : (s == 2 ? x[2] : x[3]));
  return (uint32_t)(((uint64_t)w * (uint64_t)K) >> 32);
}

// The tensor owning hash tile `tile`: the last entry with tile_begin <= tile (the host
// table lists only tensors with at least one element).
__device__ int owner_tensor(const HashTensor *tensors, int n_tensors, uint64_t tile) {
  int lo = 0, hi = n_tensors - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (tensors[mid].tile_begin <= tile) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

__global__ void __launch_bounds__(kPartThreads) hash_hist_kernel(
    const HashTensor *tensors, int n_tensors, int K, uint64_t seed, uint32_t *hist,
    unsigned long long *totals) {
  __shared__ uint32_t s_h[COPES_MAX_K];
  __shared__ int s_t;
  const uint64_t tile = blockIdx.x;
  if (threadIdx.x == 0) s_t = owner_tensor(tensors, n_tensors, tile);
  for (int k = threadIdx.x; k < K; k += kPartThreads) s_h[k] = 0;
  __syncthreads();
  const HashTensor T = tensors[s_t];
  const uint64_t e0 = (tile - T.tile_begin) * kHashTile;
  const uint64_t e1 = min(e0 + kHashTile, T.numel);
  const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  for (uint64_t e = e0 + 4ull * threadIdx.x; e < e1; e += 4ull * kPartThreads) {
    uint32_t x[4];
    const uint64_t q = e >> 2;  // e is a multiple of 4: tiles start at multiples of 16384
    philox4x32_10((uint32_t)q, (uint32_t)(q >> 32), T.tensor_id, COPES_TAG_PARTITION, k0, k1, x);
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (e + k < e1) atomicAdd(&s_h[(uint32_t)(((uint64_t)x[k] * (uint64_t)K) >> 32)], 1u);
  }
  __syncthreads();
  for (int k = threadIdx.x; k < K; k += kPartThreads) {
    hist[tile * K + k] = s_h[k];
    if (s_h[k]) atomicAdd(&totals[k], (unsigned long long)s_h[k]);
  }
}

// Block k: exclusive prefix sum over tiles of hist[tile][k] -> offsets[tile][k].
__global__ void __launch_bounds__(1024) hash_scan_kernel(const uint32_t *hist, uint64_t n_htiles,
                                                         int K, uint64_t *offsets) {
  __shared__ unsigned long long s_part[1024];
  const int k = blockIdx.x;
  const uint64_t per = (n_htiles + 1023) / 1024;
  const uint64_t t0 = min((uint64_t)threadIdx.x * per, n_htiles);
  const uint64_t t1 = min(t0 + per, n_htiles);
  unsigned long long sum = 0;
  for (uint64_t t = t0; t < t1; ++t) sum += hist[t * K + k];
  s_part[threadIdx.x] = sum;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long acc = 0;
    for (int i = 0; i < 1024; ++i) {
      const unsigned long long v = s_part[i];
      s_part[i] = acc;
      acc += v;
    }
  }
  __syncthreads();
  unsigned long long acc = s_part[threadIdx.x];
  for (uint64_t t = t0; t < t1; ++t) {
    offsets[t * K + k] = acc;
    acc += hist[t * K + k];
  }
}

struct ListTable {
  int64_t *list[COPES_MAX_K];
};

// One block per hash tile; 256 consecutive elements per step, in element order, so the
// lists come out sorted.  Within a step an element's position is its bucket's running
// offset + the counts of earlier warps + its rank among equal buckets of its warp.
__global__ void __launch_bounds__(kPartThreads) hash_scatter_kernel(
    const HashTensor *tensors, int n_tensors, int K, uint64_t seed, const uint64_t *offsets,
    const ListTable lists) {
  __shared__ unsigned long long s_run[COPES_MAX_K];
  __shared__ uint32_t s_tot[COPES_MAX_K];
  __shared__ uint32_t s_wc[kPartWarps][COPES_MAX_K];
  __shared__ int s_t;
  const uint64_t tile = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) s_t = owner_tensor(tensors, n_tensors, tile);
  for (int k = threadIdx.x; k < K; k += kPartThreads) s_run[k] = offsets[tile * K + k];
  __syncthreads();
  const HashTensor T = tensors[s_t];
  const uint64_t e0 = (tile - T.tile_begin) * kHashTile;
  const uint64_t e1 = min(e0 + kHashTile, T.numel);
  const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  const unsigned lt_mask = (1u << lane) - 1u;
  for (uint64_t step = e0; step < e1; step += kPartThreads) {
    const uint64_t e = step + threadIdx.x;
    const bool valid = e < e1;
    const uint32_t b = valid ? hash_bucket(e, T.tensor_id, k0, k1, K) : 0xFFFFFFFFu;
    for (int k = lane; k < K; k += 32) s_wc[warp][k] = 0;
    __syncwarp();
    const unsigned peers = __match_any_sync(0xffffffffu, b);
    const int rank = __popc(peers & lt_mask);
    if (valid && (__ffs(peers) - 1) == lane) s_wc[warp][b] = (uint32_t)__popc(peers);
    __syncthreads();
    for (int k = threadIdx.x; k < K; k += kPartThreads) {
      uint32_t acc = 0;
      for (int w = 0; w < kPartWarps; ++w) {
        const uint32_t c = s_wc[w][k];
        s_wc[w][k] = acc;
        acc += c;
      }
      s_tot[k] = acc;
    }
    __syncthreads();
    if (valid) lists.list[b][s_run[b] + s_wc[warp][b] + (uint32_t)rank] = (int64_t)(T.offset + e);
    __syncthreads();
    for (int k = threadIdx.x; k < K; k += kPartThreads) s_run[k] += s_tot[k];
    __syncthreads();
  }
}

// Random chunk map: chunk c has key = word 0 of Philox(seed; c, 0, CHUNK tag) and goes to
// subspace floor(rank K / n), rank = its position in (key, c) order.  The composite keys
// (key << 20) | c (c < 2^20) are distinct, so the ranks are the positions after sorting
// them: a bitonic sort over the caller's workspace (N = a power of two >= n, padded with
// the largest key), with every 4,096-key tile sorted and merged in shared memory and
// only the strides of 4,096 and more done by global-memory passes.
constexpr uint64_t kSortTile = 4096;
constexpr int kSortThreads = 512;

__global__ void __launch_bounds__(kSortThreads) chunk_keys_kernel(uint64_t n, uint64_t N, uint64_t seed,
                                                                   uint64_t *A) {
  const uint64_t i = (uint64_t)blockIdx.x * kSortThreads + threadIdx.x;
  if (i >= N) return;
  if (i < n) {
    uint32_t x[4];
    philox4x32_10((uint32_t)i, (uint32_t)(i >> 32), 0u, COPES_TAG_CHUNK, (uint32_t)seed,
                  (uint32_t)(seed >> 32), x);
    A[i] = ((uint64_t)x[0] << 20) | i;
  } else {
    A[i] = ~0ull;
  }
}

// One compare-exchange step (stage k, stride j) over a tile held in shared memory; the
// direction of each pair comes from its global index.
__device__ __forceinline__ void bitonic_smem_step(uint64_t *s, uint64_t base, uint64_t k, uint64_t j) {
  for (uint32_t t = threadIdx.x; t < kSortTile; t += kSortThreads) {
    const uint32_t l = t ^ (uint32_t)j;
    if (l > t) {
      const bool up = ((base + t) & k) == 0;
      const uint64_t a = s[t], b = s[l];
      if ((a > b) == up) {
        s[t] = b;
        s[l] = a;
      }
    }
  }
  __syncthreads();
}

// k_stage == 0: sort every tile (stages 2 .. kSortTile).  Otherwise: the strides below
// kSortTile of stage k_stage.
__global__ void __launch_bounds__(kSortThreads) bitonic_tile_kernel(uint64_t *A, uint64_t k_stage) {
  __shared__ uint64_t s[kSortTile];
  const uint64_t base = (uint64_t)blockIdx.x * kSortTile;
  for (uint32_t t = threadIdx.x; t < kSortTile; t += kSortThreads) s[t] = A[base + t];
  __syncthreads();
  if (k_stage == 0) {
    for (uint64_t k = 2; k <= kSortTile; k <<= 1)
      for (uint64_t j = k >> 1; j > 0; j >>= 1) bitonic_smem_step(s, base, k, j);
  } else {
    for (uint64_t j = kSortTile >> 1; j > 0; j >>= 1) bitonic_smem_step(s, base, k_stage, j);
  }
  for (uint32_t t = threadIdx.x; t < kSortTile; t += kSortThreads) A[base + t] = s[t];
}

__global__ void __launch_bounds__(kSortThreads) bitonic_global_kernel(uint64_t *A, uint64_t N, uint64_t j,
                                                                      uint64_t k) {
  const uint64_t i = (uint64_t)blockIdx.x * kSortThreads + threadIdx.x;
  if (i >= N) return;
  const uint64_t l = i ^ j;
  if (l > i) {
    const bool up = (i & k) == 0;
    const uint64_t a = A[i], b = A[l];
    if ((a > b) == up) {
      A[i] = b;
      A[l] = a;
    }
  }
}

__global__ void __launch_bounds__(kSortThreads) chunk_map_kernel(const uint64_t *A, uint64_t n, int K,
                                                                 uint32_t *map) {
  const uint64_t i = (uint64_t)blockIdx.x * kSortThreads + threadIdx.x;
  if (i >= n) return;
  map[A[i] & 0xFFFFFull] = (uint32_t)((i * (uint64_t)K) / n);
}

uint64_t chunk_sort_size(uint64_t n_chunks) {
  uint64_t N = kSortTile;
  while (N < n_chunks) N <<= 1;
  return N;
}

cudaError_t launch_hash_hist(const HashTensor *tensors, int n_tensors, uint64_t n_htiles, int K,
                             uint64_t seed, uint32_t *hist, unsigned long long *totals,
                             cudaStream_t s) {
  if (n_htiles == 0) return cudaSuccess;
  hash_hist_kernel<<<(unsigned)n_htiles, kPartThreads, 0, s>>>(tensors, n_tensors, K, seed, hist,
                                                                totals);
  return cudaGetLastError();
}

cudaError_t launch_hash_scan(const uint32_t *hist, uint64_t n_htiles, int K, uint64_t *offsets,
                             cudaStream_t s) {
  if (n_htiles == 0) return cudaSuccess;
  hash_scan_kernel<<<K, 1024, 0, s>>>(hist, n_htiles, K, offsets);
  return cudaGetLastError();
}

cudaError_t launch_hash_scatter(const HashTensor *tensors, int n_tensors, uint64_t n_htiles,
                                int K, uint64_t seed, const uint64_t *offsets,
                                int64_t *const *lists, cudaStream_t s) {
  if (n_htiles == 0) return cudaSuccess;
  ListTable t;
  for (int k = 0; k < COPES_MAX_K; ++k) t.list[k] = k < K ? lists[k] : nullptr;
  hash_scatter_kernel<<<(unsigned)n_htiles, kPartThreads, 0, s>>>(tensors, n_tensors, K, seed,
                                                                   offsets, t);
  return cudaGetLastError();
}

cudaError_t launch_random_chunk_map(uint64_t n_chunks, int K, uint64_t seed, uint32_t *map,
                                    uint64_t *keys, cudaStream_t s) {
  const uint64_t N = chunk_sort_size(n_chunks);
  const unsigned gblocks = (unsigned)((N + kSortThreads - 1) / kSortThreads);
  const unsigned tiles = (unsigned)(N / kSortTile);
  chunk_keys_kernel<<<gblocks, kSortThreads, 0, s>>>(n_chunks, N, seed, keys);
  bitonic_tile_kernel<<<tiles, kSortThreads, 0, s>>>(keys, 0);
  for (uint64_t k = 2 * kSortTile; k <= N; k <<= 1) {
    for (uint64_t j = k >> 1; j >= kSortTile; j >>= 1)
      bitonic_global_kernel<<<gblocks, kSortThreads, 0, s>>>(keys, N, j, k);
    bitonic_tile_kernel<<<tiles, kSortThreads, 0, s>>>(keys, k);
  }
  const unsigned mblocks = (unsigned)((n_chunks + kSortThreads - 1) / kSortThreads);
  chunk_map_kernel<<<mblocks, kSortThreads, 0, s>>>(keys, n_chunks, K, map);
  return cudaGetLastError();
}

// Tile table of a list of disjoint ranges, written on the device: tile t lies in the range
// r with first[r] <= t < first[r + 1] and covers [begin[r] + (t - first[r]) tile_size,
// min(that + tile_size, end[r])).  The ranges travel in the launch's parameters, so no
// host staging of the table is needed.
__global__ void __launch_bounds__(256) tile_expand_kernel(const __grid_constant__ TileRanges a, uint64_t *tiles) {
  for (uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; t < a.first[a.n_ranges];
       t += (uint64_t)gridDim.x * blockDim.x) {
    int lo = 0, hi = a.n_ranges - 1;  // the last range whose first tile is <= t
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (a.first[mid] <= t) lo = mid;
      else hi = mid - 1;
    }
    const uint64_t b = a.begin[lo] + (t - a.first[lo]) * a.tile_size;
    const uint64_t e = min(b + a.tile_size, a.end[lo]);
    reinterpret_cast<ulonglong2 *>(tiles)[t] = make_ulonglong2(b, e);
  }
}

cudaError_t launch_tile_expand(const TileRanges &r, uint64_t *tiles, cudaStream_t s) {
  const uint64_t n = r.first[r.n_ranges];
  if (n == 0) return cudaSuccess;
  const uint64_t want = (n + 255) / 256;
  const unsigned blocks = (unsigned)(want < 4096 ? want : 4096);
  tile_expand_kernel<<<blocks, 256, 0, s>>>(r, tiles);
  return cudaGetLastError();
}

unsigned read_and_clear_partition_errors() {
  unsigned v = 0, zero = 0;
  cudaMemcpyFromSymbol(&v, g_partition_error, sizeof(v));
  if (v) cudaMemcpyToSymbol(g_partition_error, &zero, sizeof(zero));
  return v;
}

}  // namespace copes
