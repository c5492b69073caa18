// Partition replay (Supp. A.8 "Partition Replay"; Eq. 7): the ES kernels over subspace k
// of the hash partition (K, seed) with membership recomputed from the partition seed, not
// read from a stored index list.  Each block takes 4 consecutive 16,384-element hash
// tiles; each warp streams through its 2,048-element stretch of every tile (replay_stream):
//  - it hashes 32 four-element groups at a time -- one Philox4x32-10 call per group at
//    counter (e >> 2, tensor id, TAG_PARTITION), bucket floor(x K / 2^32) per word, or,
//    when the subspace carries a membership mask built once per visit, reads their bits --
//    and appends the members of subspace k to its shared-memory buffer;
//  - whenever the buffer holds a full batch, the warp processes it one member per lane,
//    exactly as the gather kernels process an index list: perturb / restore / commit /
//    init, or the fused update regenerating the P normals of each element.
// Every element's arithmetic is that of the gather path, so the results are identical to
// those over the INDICES list of (K, seed, k).
#include <type_traits>

#include "es_common.cuh"

namespace copes {

__device__ unsigned int g_replay_error = 0;

__device__ __forceinline__ void replay_flag(unsigned bit) { atomicOr(&g_replay_error, bit); }

constexpr int kReplayTile = (int)kHashTile;  // elements per hash tile
constexpr int kReplayTilesPerBlock = 4;      // consecutive hash tiles per block
static_assert(kReplayTile % 4 == 0 && kReplayTile <= 65536, "tile offsets fit 16 bits");
constexpr int kReplayWarpGroups = kReplayTile / 4 / (kThreads / 32);  // groups per warp per tile
constexpr int kReplayIters = kReplayWarpGroups / 32;                  // 32 groups per iteration

constexpr uint64_t kMaskWordsPerTile = kReplayTile / 32;  // membership mask: one bit per element

struct ReplayTile {
  uint64_t g0;        // global index of the tile's first element
  uint64_t q0;        // partition counter of the tile's first group (tensor-local e >> 2)
  uint32_t len;       // elements in the tile (0: skip the tile)
  uint32_t tensor_id;
};

// Hash tile `tile`: its tensor comes from the table's tile map; every thread reads the
// same entries (cached broadcasts), so the result is block-uniform.  A tile the table
// maps outside its tensor or past the arena is skipped and flagged.
__device__ __forceinline__ ReplayTile replay_tile(const ReplayArgs &r, uint64_t n_alloc, uint64_t tile) {
  ReplayTile t{};
  const uint32_t ti = r.tile_tensor[tile];
  if (ti >= (uint32_t)r.n_tensors) {
    if (threadIdx.x == 0) replay_flag(kErrPartition);
    return t;
  }
  const HashTensor T = r.table[ti];
  const uint64_t e0 = (tile - T.tile_begin) * (uint64_t)kReplayTile;
  if (tile < T.tile_begin || e0 >= T.numel) {
    if (threadIdx.x == 0) replay_flag(kErrPartition);
    return t;
  }
  const uint32_t len = (uint32_t)min((uint64_t)kReplayTile, T.numel - e0);
  const uint64_t g0 = T.offset + e0;
  if (g0 + len > n_alloc || (g0 & 3ull) != 0) {
    if (threadIdx.x == 0) replay_flag(kErrIndexRange);
    return t;
  }
  t.g0 = g0;
  t.q0 = e0 >> 2;
  t.len = len;
  t.tensor_id = T.tensor_id;
  return t;
}

// Warp-streamed replay over the block's hash tiles.  Each warp owns a 2,048-element
// stretch of every tile and walks it 32 groups (one per lane) at a time: it hashes the
// groups, appends the members of subspace r.k to its shared-memory buffer with one ballot
// per word slot, and whenever the buffer holds BATCH members it processes them, BATCH / 32
// per lane, every lane busy, so the hashing (ALU) interleaves with the members' scattered
// loads and stores.  The warps' leftovers (fewer than BATCH each) are pooled and processed
// by the whole block at the end; `flush` then runs once.  Every warp runs the same
// iterations, so the full-warp ballots and shuffles see all 32 lanes.  MASK: membership
// comes from r.mask (non-null) instead of the hash; a compile-time choice, so the hashing
// variant carries no mask code.
template <int BATCH, bool MASK, typename Fn, typename Flush>
__device__ __forceinline__ void replay_stream(const ReplayArgs &r, uint64_t n_alloc, uint32_t *wbuf,
                                              uint64_t (*s_g0)[kReplayTilesPerBlock], uint32_t *pool,
                                              int *pool_n, Fn process, Flush flush) {
  constexpr int U = BATCH / 32;
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t warp = threadIdx.x >> 5;
  const uint64_t t_first = (uint64_t)blockIdx.x * kReplayTilesPerBlock;
  const uint64_t t_end = min(t_first + kReplayTilesPerBlock, r.n_tiles);
  // buffer entries are (tile within the block) << 16 | (offset within the tile); each warp
  // keeps the tiles' first global indices in its own row of s_g0
  uint64_t *wg0 = s_g0[warp];
  auto global = [&](uint32_t e) { return wg0[e >> 16] + (e & 0xFFFFu); };
  const uint32_t lt = (1u << lane) - 1u;  // lanes below this one
  int pending = 0;  // warp-uniform
  // One iteration: the warp hashes 32 groups (128 elements, one group per lane) and
  // appends their members with one ballot per word slot; FULL drops the tile-end check.
  auto iteration = [&](const ReplayTile &t, uint64_t tile, uint32_t tag, uint32_t q_lo0, uint32_t q_hi,
                       uint32_t e, auto full) {
    bool m[4];  // membership of the group's 4 elements
    if constexpr (MASK) {
      const uint32_t nib = r.mask[tile * kMaskWordsPerTile + (e >> 5)] >> (e & 31u);
#pragma unroll
      for (int i = 0; i < 4; ++i) m[i] = (nib >> i) & 1u;
    } else {
      uint32_t x[4];
      philox4x32_10_rk(q_lo0 + (e >> 2), q_hi, t.tensor_id, COPES_TAG_PARTITION, r.rk, x);
#pragma unroll
      for (int i = 0; i < 4; ++i)
        // floor(x K / 2^32) == k  <=>  x - lo <= span in 32-bit unsigned arithmetic
        m[i] = x[i] - r.lo <= r.span && (decltype(full)::value || e + i < t.len);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t bal = __ballot_sync(0xffffffffu, m[i]);
      if (m[i]) wbuf[pending + __popc(bal & lt)] = tag | (e + i);
      pending += __popc(bal);
    }
    __syncwarp();
    while (pending >= BATCH) {  // take the newest BATCH entries
      uint64_t g[U];
      bool ok[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        g[u] = global(wbuf[pending - BATCH + u * 32 + lane]);
        ok[u] = true;
      }
      __syncwarp();  // read before the next append overwrites these slots
      pending -= BATCH;
      process(g, ok);
    }
  };
  for (uint64_t tile = t_first; tile < t_end; ++tile) {
    const ReplayTile t = replay_tile(r, n_alloc, tile);
    const uint32_t tag = (uint32_t)(tile - t_first) << 16;
    // q0 is a multiple of 4096 and the tile has 4096 groups, so q0 + group never carries
    // out of 32 bits
    const uint32_t q_lo0 = (uint32_t)t.q0, q_hi = (uint32_t)(t.q0 >> 32);
    if (lane == 0) wg0[tile - t_first] = t.g0;
    __syncwarp();
    const uint32_t e0 = warp * (4u * kReplayWarpGroups) + 4u * lane;  // this lane's first group
    if (t.len == (uint32_t)kReplayTile) {
      for (int it = 0; it < kReplayIters; ++it)
        iteration(t, tile, tag, q_lo0, q_hi, e0 + 128u * it, std::true_type{});
    } else if (t.len > 0) {
      for (int it = 0; it < kReplayIters; ++it)
        iteration(t, tile, tag, q_lo0, q_hi, e0 + 128u * it, std::false_type{});
    }
  }
  // pool the leftovers and process them with the whole block
  int at = 0;
  if (lane == 0 && pending) at = atomicAdd(pool_n, pending);
  at = __shfl_sync(0xffffffffu, at, 0);
  for (int p = lane; p < pending; p += 32) pool[at + p] = wbuf[p];
  __syncthreads();
  const int n = *pool_n;
  wg0 = s_g0[0];  // every warp recorded the same tiles
  for (int p0 = threadIdx.x; p0 < n; p0 += kThreads * U) {
    uint64_t g[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int p = p0 + kThreads * u;
      ok[u] = p < n;
      g[u] = ok[u] ? global(pool[p]) : wg0[0];
    }
    process(g, ok);
  }
  flush();
}

template <int OP>
constexpr uint32_t replay_tag() { return OP == kOpInit ? COPES_TAG_INIT : COPES_TAG_NOISE; }

// Perturb / restore / commit / init over the members of the block's hash tiles: four
// members per lane per batch, their master loads issued together.
template <int OP, typename WT, bool MASK>
__global__ void __launch_bounds__(kThreads) replay_elem_kernel(const __grid_constant__ ElemArgs a,
                                                               const __grid_constant__ ReplayArgs r) {
  constexpr int BATCH = 128;
  constexpr int U = BATCH / 32;
  __shared__ uint32_t s_buf[kThreads / 32][BATCH + 128];
  __shared__ uint32_t s_pool[(kThreads / 32) * BATCH];
  __shared__ uint64_t s_g0[kThreads / 32][kReplayTilesPerBlock];
  __shared__ int s_pool_n;
  if (threadIdx.x == 0) s_pool_n = 0;
  __syncthreads();
  float *__restrict__ master = a.master;
  replay_stream<BATCH, MASK>(r, a.n_alloc, s_buf[threadIdx.x >> 5], s_g0, s_pool, &s_pool_n,
                             [&](const uint64_t (&g)[U], const bool (&ok_in)[U]) {
    bool ok[U];
    float th[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      ok[u] = ok_in[u];
      if ((OP == kOpPerturbPair || OP == kOpPartner) && ok[u] &&
          (g[u] < a.partner_base || g[u] - a.partner_base >= a.partner_len)) {
        replay_flag(kErrPartnerRange);
        ok[u] = false;
      }
      th[u] = (OP != kOpInit && OP != kOpPartner && ok[u]) ? master[g[u]] : 0.0f;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      if constexpr (OP == kOpPartner) {
        reinterpret_cast<WT *>(a.w)[g[u]] = reinterpret_cast<const WT *>(a.partner)[g[u] - a.partner_base];
        continue;
      }
      float v, vp = 0.0f;
      if (OP == kOpRestore) {
        v = th[u];
      } else {
        uint32_t x[4];
        const uint64_t q = g[u] >> 2;
        philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, replay_tag<OP>(), a.rk, x);
        const uint32_t sel = (uint32_t)g[u] & 3u;
        const uint32_t wd = sel == 0 ? x[0] : (sel == 1 ? x[1] : (sel == 2 ? x[2] : x[3]));
        float xv, r;
        normal_parts(wd, a.coeffs.central, a.coeffs.tail, xv, r);  // r = a * R(L)
        v = __fmaf_rn(r, xv, OP == kOpInit ? a.b : th[u]);
        if (OP == kOpPerturbPair) vp = __fmaf_rn(-r, xv, th[u]);
        if (OP == kOpInit) master[g[u]] = v;
      }
      WStore<WT>::one(a.w, g[u], v);
      if (OP == kOpRestore || OP == kOpInit) store_copies_one<WT>(a.copies, g[u], v);
      if (OP == kOpPerturbPair) WStore<WT>::one(a.partner, g[u] - a.partner_base, vp);
    }
  }, [] {});
}

// The fused update over the members of the block's hash tiles: two members per lane per
// batch, each regenerating the P normals of its element.
template <typename WT, bool COMMIT, bool MASK>
__global__ void __launch_bounds__(kThreads) replay_update_kernel(const __grid_constant__ UpdateArgs a,
                                                                 const __grid_constant__ ReplayArgs r) {
  constexpr int BATCH = 64;
  constexpr int U = BATCH / 32;
  __shared__ float s_w[COPES_MAX_NOISE];
  __shared__ __align__(16) uint32_t s_rk[COPES_MAX_NOISE][20];
  __shared__ uint32_t s_buf[kThreads / 32][BATCH + 128];
  __shared__ uint32_t s_pool[(kThreads / 32) * BATCH];
  __shared__ uint64_t s_g0[kThreads / 32][kReplayTilesPerBlock];
  __shared__ int s_pool_n;
  if (threadIdx.x == 0) s_pool_n = 0;
  noise_weights_to_smem(a, s_w, s_rk);  // ends with __syncthreads
  float *__restrict__ master = a.master;
  const int P = a.n_noise;
  replay_stream<BATCH, MASK>(r, a.n_alloc, s_buf[threadIdx.x >> 5], s_g0, s_pool, &s_pool_n,
                             [&](const uint64_t (&g)[U], const bool (&ok)[U]) {
    float acc[U];
#pragma unroll
    for (int u = 0; u < U; ++u) acc[u] = 0.0f;
    for (int j = 0; j < P; ++j) {
      uint32_t rk[20];
#pragma unroll
      for (int q = 0; q < 20; q += 4) {
        const uint4 v = *reinterpret_cast<const uint4 *>(&s_rk[j][q]);
        rk[q] = v.x, rk[q + 1] = v.y, rk[q + 2] = v.z, rk[q + 3] = v.w;
      }
      const float wj = s_w[j];
      uint32_t wd[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        uint32_t x[4];
        const uint64_t q = g[u] >> 2;
        philox4x32_10_rk((uint32_t)q, (uint32_t)(q >> 32), 0u, COPES_TAG_NOISE, rk, x);
        const uint32_t sel = (uint32_t)g[u] & 3u;
        wd[u] = sel == 0 ? x[0] : (sel == 1 ? x[1] : (sel == 2 ? x[2] : x[3]));
      }
      // the two members' normals as one packed pair (bit-identical to one at a time)
      static_assert(U == 2, "normals are paired");
      float eps0, eps1;
      normal_pair_x2(wd[0], wd[1], eps0, eps1);
      acc[0] = __fmaf_rn(wj, eps0, acc[0]);
      acc[1] = __fmaf_rn(wj, eps1, acc[1]);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      const float v = __fmaf_rn(a.coef, acc[u], master[g[u]]);
      master[g[u]] = v;
      if (COMMIT) {
        WStore<WT>::one(a.w, g[u], v);
        store_copies_one<WT>(a.copies, g[u], v);
      }
    }
  }, [] {});
}

static unsigned replay_blocks(uint64_t n_tiles) {
  return (unsigned)((n_tiles + kReplayTilesPerBlock - 1) / kReplayTilesPerBlock);
}

// Membership mask of subspace r.k: bit (e mod 32) of word tile * 512 + e / 32 is set when
// element e of hash tile `tile` belongs to it.  One block per hash tile; each lane hashes
// one group per step and 8 lanes' 4-bit nibbles make a word.  Tiles the table maps outside
// the arena are flagged and written as empty.
__global__ void __launch_bounds__(kThreads) replay_mask_kernel(const __grid_constant__ ReplayArgs r,
                                                               uint64_t n_alloc, uint32_t *mask) {
  const uint64_t tile = blockIdx.x;
  const ReplayTile t = replay_tile(r, n_alloc, tile);
  const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
  const uint32_t q_lo0 = (uint32_t)t.q0, q_hi = (uint32_t)(t.q0 >> 32);
  for (int it = 0; it < kReplayIters; ++it) {
    const uint32_t e = warp * (4u * kReplayWarpGroups) + 128u * it + 4u * lane;
    uint32_t nib = 0;
    if (e < t.len) {
      uint32_t x[4];
      philox4x32_10_rk(q_lo0 + (e >> 2), q_hi, t.tensor_id, COPES_TAG_PARTITION, r.rk, x);
#pragma unroll
      for (int i = 0; i < 4; ++i)
        nib |= (x[i] - r.lo <= r.span && e + i < t.len) ? (1u << i) : 0u;
    }
    uint32_t word = nib << (4u * (lane & 7u));
    word |= __shfl_xor_sync(0xffffffffu, word, 1);
    word |= __shfl_xor_sync(0xffffffffu, word, 2);
    word |= __shfl_xor_sync(0xffffffffu, word, 4);
    if ((lane & 7u) == 0) mask[tile * kMaskWordsPerTile + (e >> 5)] = word;
  }
}

cudaError_t launch_replay_mask(const ReplayArgs &r, uint64_t n_alloc, uint32_t *mask, cudaStream_t s) {
  if (r.n_tiles == 0) return cudaSuccess;
  replay_mask_kernel<<<(unsigned)r.n_tiles, kThreads, 0, s>>>(r, n_alloc, mask);
  return cudaGetLastError();
}

template <int OP, typename WT>
static cudaError_t launch_replay_elem_typed(const ElemArgs &a, const ReplayArgs &r, cudaStream_t s) {
  if (r.n_tiles == 0) return cudaSuccess;
  if (r.mask)
    replay_elem_kernel<OP, WT, true><<<replay_blocks(r.n_tiles), kThreads, 0, s>>>(a, r);
  else
    replay_elem_kernel<OP, WT, false><<<replay_blocks(r.n_tiles), kThreads, 0, s>>>(a, r);
  return cudaGetLastError();
}

template <typename WT>
static cudaError_t launch_replay_elem_dtype(int op, const ElemArgs &a, const ReplayArgs &r,
                                            cudaStream_t s) {
  switch (op) {
    case kOpPerturb: return launch_replay_elem_typed<kOpPerturb, WT>(a, r, s);
    case kOpRestore: return launch_replay_elem_typed<kOpRestore, WT>(a, r, s);
    case kOpPerturbPair: return launch_replay_elem_typed<kOpPerturbPair, WT>(a, r, s);
    case kOpPartner: return launch_replay_elem_typed<kOpPartner, WT>(a, r, s);
    case kOpInit: return launch_replay_elem_typed<kOpInit, WT>(a, r, s);
    default: return cudaErrorInvalidValue;  // the other ops have no replay form
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
  if (r.mask)
    replay_update_kernel<WT, COMMIT, true><<<replay_blocks(r.n_tiles), kThreads, 0, s>>>(a, r);
  else
    replay_update_kernel<WT, COMMIT, false><<<replay_blocks(r.n_tiles), kThreads, 0, s>>>(a, r);
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
