// Partition replay (Supp. A.8 "Partition Replay"; Eq. 7): the ES kernels over subspace k
// of the hash partition (K, seed) with membership recomputed from the partition seed, not
// read from a stored index list.  One block per 16,384-element hash tile of one tensor:
//  phase 1  every thread hashes its 4-element groups -- one Philox4x32-10 call per group
//           at counter (e >> 2, tensor id, TAG_PARTITION), bucket floor(x K / 2^32) per
//           word -- and appends the tile offsets of the members of subspace k to a list
//           in shared memory (warp-aggregated appends; the list order is arbitrary);
//  phase 2  the block works through the list exactly as the gather kernels work through
//           an index list: perturb / restore / commit / init one element per thread, or
//           the fused update regenerating the P normals of each element.
// Every element's arithmetic is that of the gather path, so the results are identical to
// those over the INDICES list of (K, seed, k).
#include "es_common.cuh"

namespace copes {

__device__ unsigned int g_replay_error = 0;

__device__ __forceinline__ void replay_flag(unsigned bit) { atomicOr(&g_replay_error, bit); }

constexpr int kReplayTile = (int)kHashTile;  // elements per block
static_assert(kReplayTile % 4 == 0 && kReplayTile <= 65536, "tile offsets are stored as uint16");

struct ReplayTile {
  uint64_t g0;        // global index of the tile's first element
  uint64_t q0;        // partition counter of the tile's first group (tensor-local e >> 2)
  uint32_t len;       // elements in the tile (0: skip the tile)
  uint32_t tensor_id;
};

// The tile's tensor and extent.  Thread 0 searches the table; the result is broadcast
// through shared memory.  A tile outside its tensor or past the arena is skipped and
// flagged.
__device__ __forceinline__ void replay_locate(const ReplayArgs &r, uint64_t n_alloc, ReplayTile *s_tile,
                                              int *s_n) {
  if (threadIdx.x == 0) {
    const uint64_t tile = blockIdx.x;
    int lo = 0, hi = r.n_tensors - 1;  // last entry with tile_begin <= tile
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (r.table[mid].tile_begin <= tile) lo = mid;
      else hi = mid - 1;
    }
    const HashTensor T = r.table[lo];
    ReplayTile t{};
    const uint64_t e0 = (tile - T.tile_begin) * (uint64_t)kReplayTile;
    if (tile < T.tile_begin || e0 >= T.numel) {
      replay_flag(kErrPartition);
    } else {
      t.len = (uint32_t)min((uint64_t)kReplayTile, T.numel - e0);
      t.g0 = T.offset + e0;
      t.q0 = e0 >> 2;
      t.tensor_id = T.tensor_id;
      if (t.g0 + t.len > n_alloc || (t.g0 & 3ull) != 0) {
        replay_flag(kErrIndexRange);
        t.len = 0;
      }
    }
    *s_tile = t;
    *s_n = 0;
  }
  __syncthreads();
}

// Phase 1: the tile offsets of the members of subspace r.k, appended to s_list; returns
// their number.  Every warp runs the same number of iterations, so the full-warp
// shuffles below see all 32 lanes.
__device__ __forceinline__ int replay_members(const ReplayArgs &r, const ReplayTile &t,
                                              uint16_t *s_list, int *s_n) {
  uint32_t rk[20];
  philox_round_keys(r.seed_lo, r.seed_hi, rk);
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t n_groups = (t.len + 3u) / 4u;
  for (uint32_t base = 0; base < n_groups; base += kThreads) {
    const uint32_t grp = base + threadIdx.x;
    uint32_t mask = 0;
    if (grp < n_groups) {
      const uint64_t q = t.q0 + grp;
      uint32_t x[4];
      philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), t.tensor_id, COPES_TAG_PARTITION, rk, x);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t bucket = (uint32_t)(((uint64_t)x[i] * (uint64_t)r.K) >> 32);
        if (4u * grp + i < t.len && bucket == (uint32_t)r.k) mask |= 1u << i;
      }
    }
    const int c = __popc(mask);
    int incl = c;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= (uint32_t)d) incl += y;
    }
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    int wbase = 0;
    if (lane == 31 && total) wbase = atomicAdd(s_n, total);
    wbase = __shfl_sync(0xffffffffu, wbase, 31);
    int pos = wbase + incl - c;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (mask & (1u << i)) s_list[pos++] = (uint16_t)(4u * grp + i);
  }
  __syncthreads();
  return *s_n;
}

template <int OP>
constexpr uint32_t replay_tag() { return OP == kOpInit ? COPES_TAG_INIT : COPES_TAG_NOISE; }

// Perturb / restore / commit / init over the members of one hash tile.
template <int OP, typename WT>
__global__ void __launch_bounds__(kThreads) replay_elem_kernel(const ElemArgs a, const ReplayArgs r) {
  __shared__ __align__(16) uint16_t s_list[kReplayTile];
  __shared__ ReplayTile s_tile;
  __shared__ int s_n;
  replay_locate(r, a.n_alloc, &s_tile, &s_n);
  const ReplayTile t = s_tile;
  const int n = replay_members(r, t, s_list, &s_n);
  float *__restrict__ master = a.master;
  for (int p = threadIdx.x; p < n; p += kThreads) {
    const uint64_t g = t.g0 + s_list[p];
    float v;
    if (OP == kOpRestore) {
      v = master[g];
    } else {
      uint32_t x[4];
      const uint64_t q = g >> 2;
      philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, replay_tag<OP>(), a.rk, x);
      const uint32_t sel = (uint32_t)g & 3u;
      const uint32_t wd = sel == 0 ? x[0] : (sel == 1 ? x[1] : (sel == 2 ? x[2] : x[3]));
      v = scaled_normal_plus(wd, a.coeffs, OP == kOpPerturb ? master[g] : a.b);
      if (OP == kOpInit) master[g] = v;
    }
    WStore<WT>::one(a.w, g, v);
  }
}

// The fused update over the members of one hash tile.  Dynamic shared memory holds the
// noise vectors' round keys [P][20], their weights [P] and the member list.
template <typename WT, bool COMMIT>
__global__ void __launch_bounds__(kThreads) replay_update_kernel(const __grid_constant__ UpdateArgs a,
                                                                 const ReplayArgs r) {
  extern __shared__ __align__(16) unsigned char smem[];
  auto *s_rk = reinterpret_cast<uint32_t (*)[20]>(smem);
  float *s_w = reinterpret_cast<float *>(smem + (size_t)a.n_noise * 80);
  uint16_t *s_list = reinterpret_cast<uint16_t *>(smem + (size_t)a.n_noise * 84);
  __shared__ ReplayTile s_tile;
  __shared__ int s_n;
  noise_weights_to_smem(a, s_w, s_rk);
  replay_locate(r, a.n_alloc, &s_tile, &s_n);
  const ReplayTile t = s_tile;
  const int n = replay_members(r, t, s_list, &s_n);
  constexpr int U = 2;
  float *__restrict__ master = a.master;
  const int P = a.n_noise;
  for (int p0 = threadIdx.x; p0 < n; p0 += kThreads * U) {
    uint64_t g[U];
    float acc[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int p = p0 + kThreads * u;
      ok[u] = p < n;
      g[u] = t.g0 + (ok[u] ? s_list[p] : 0);
      acc[u] = 0.0f;
    }
    for (int j = 0; j < P; ++j) {
      uint32_t rk[20];
#pragma unroll
      for (int q = 0; q < 20; q += 4) {
        const uint4 v = *reinterpret_cast<const uint4 *>(&s_rk[j][q]);
        rk[q] = v.x, rk[q + 1] = v.y, rk[q + 2] = v.z, rk[q + 3] = v.w;
      }
      const float wj = s_w[j];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        uint32_t x[4];
        const uint64_t q = g[u] >> 2;
        philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, COPES_TAG_NOISE, rk, x);
        const uint32_t sel = (uint32_t)g[u] & 3u;
        const uint32_t wd = sel == 0 ? x[0] : (sel == 1 ? x[1] : (sel == 2 ? x[2] : x[3]));
        acc[u] = __fmaf_rn(wj, normal_from_word(wd), acc[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      const float v = __fmaf_rn(a.coef, acc[u], master[g[u]]);
      master[g[u]] = v;
      if (COMMIT) WStore<WT>::one(a.w, g[u], v);
    }
  }
}

template <int OP, typename WT>
static cudaError_t launch_replay_elem_typed(const ElemArgs &a, const ReplayArgs &r, cudaStream_t s) {
  if (r.n_tiles == 0) return cudaSuccess;
  replay_elem_kernel<OP, WT><<<(unsigned)r.n_tiles, kThreads, 0, s>>>(a, r);
  return cudaGetLastError();
}

template <typename WT>
static cudaError_t launch_replay_elem_dtype(int op, const ElemArgs &a, const ReplayArgs &r,
                                            cudaStream_t s) {
  switch (op) {
    case kOpPerturb: return launch_replay_elem_typed<kOpPerturb, WT>(a, r, s);
    case kOpRestore: return launch_replay_elem_typed<kOpRestore, WT>(a, r, s);
    default: return launch_replay_elem_typed<kOpInit, WT>(a, r, s);
  }
}

cudaError_t launch_replay_elementwise(int op, int dtype, const ElemArgs &a, const ReplayArgs &r,
                                      cudaStream_t s) {
  return dtype == COPES_BF16 ? launch_replay_elem_dtype<__nv_bfloat16>(op, a, r, s)
                             : launch_replay_elem_dtype<float>(op, a, r, s);
}

template <typename WT, bool COMMIT>
static cudaError_t launch_replay_update_typed(const UpdateArgs &a, const ReplayArgs &r, cudaStream_t s) {
  if (r.n_tiles == 0) return cudaSuccess;
  const size_t smem = (size_t)a.n_noise * 84 + (size_t)kReplayTile * 2;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(replay_update_kernel<WT, COMMIT>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  replay_update_kernel<WT, COMMIT><<<(unsigned)r.n_tiles, kThreads, smem, s>>>(a, r);
  return cudaGetLastError();
}

cudaError_t launch_replay_update(int dtype, const UpdateArgs &a, const ReplayArgs &r, cudaStream_t s) {
  if (dtype == COPES_BF16)
    return a.fuse_commit ? launch_replay_update_typed<__nv_bfloat16, true>(a, r, s)
                         : launch_replay_update_typed<__nv_bfloat16, false>(a, r, s);
  return a.fuse_commit ? launch_replay_update_typed<float, true>(a, r, s)
                       : launch_replay_update_typed<float, false>(a, r, s);
}

unsigned read_and_clear_replay_errors() {
  unsigned v = 0, zero = 0;
  cudaMemcpyFromSymbol(&v, g_replay_error, sizeof(v));
  if (v) cudaMemcpyToSymbol(g_replay_error, &zero, sizeof(zero));
  return v;
}

}  // namespace copes
