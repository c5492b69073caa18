// CPU weight backup mode (Supp. A.8 "CPU Weight Backup"): bf16 working weights in HBM and
// the shared context as a bf16 copy in pinned host memory, read and written by the
// kernels directly over the host link.  Tile subspaces; 4-element groups are one Philox
// counter and one 8-byte load or store of each bf16 array.
//  save     backup[g] = w[g]
//  perturb  w[g] = round(fma(s sigma, eps[g], backup[g]))      (Eq. 8)
//  pair     perturb, and partner[g - base] = round(fma(-s sigma, eps[g], backup[g]))
//  restore  w[g] = backup[g]
//  update   t = fma(coef, sum_j w_j eps_j[g], backup[g]);  w[g] = backup[g] = round(t)
// The perturb and update arithmetic is that of the master path with theta = backup.
#include "es_common.cuh"

namespace copes {

__device__ unsigned int g_backup_error = 0;

__device__ __forceinline__ void backup_flag(unsigned bit) { atomicOr(&g_backup_error, bit); }

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

__device__ __forceinline__ void unpack4(uint2 v, float t[4]) {
  t[0] = __uint_as_float(v.x << 16);
  t[1] = __uint_as_float(v.x & 0xFFFF0000u);
  t[2] = __uint_as_float(v.y << 16);
  t[3] = __uint_as_float(v.y & 0xFFFF0000u);
}

__device__ __forceinline__ uint2 pack4(const float v[4]) {
  return make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
}

// Validated tile bounds: false (and a flag) for a tile outside the arena.
__device__ __forceinline__ bool backup_tile(const uint64_t *tiles, uint64_t t, uint64_t n_alloc,
                                            uint64_t &b, uint64_t &e) {
  b = tiles[2 * t];
  e = tiles[2 * t + 1];
  if (b > e || e > n_alloc || e - b > (uint64_t)COPES_TILE_MAX) {
    if (threadIdx.x == 0) backup_flag(kErrTileRange);
    return false;
  }
  return true;
}

// One block per tile; thread-strided 4-element groups.
template <int OP>
__global__ void __launch_bounds__(kThreads) backup_elem_kernel(const __grid_constant__ ElemArgs a,
                                                               uint16_t *backup) {
  uint64_t b, e;
  if (!backup_tile(a.tiles, blockIdx.x, a.n_alloc, b, e)) return;
  if (OP == kBackupPerturbPair && (b < a.partner_base || e - a.partner_base > a.partner_len)) {
    if (threadIdx.x == 0) backup_flag(kErrPartnerRange);
    return;
  }
  constexpr bool kPerturb = OP == kBackupPerturb || OP == kBackupPerturbPair;
  uint16_t *w = static_cast<uint16_t *>(a.w);
  // partner element g at pw[g - partner_base]; partner_base is a multiple of 4 and at most b,
  // so every group of the tile starts at or after it
  uint16_t *pw = static_cast<uint16_t *>(a.partner);
  const uint16_t *src = OP == kBackupSave ? w : backup;
  uint16_t *dst = OP == kBackupSave ? backup : w;
  for (uint64_t g4 = (b & ~3ull) + 4ull * threadIdx.x; g4 < e; g4 += 4ull * kThreads) {
    const bool full = g4 >= b && g4 + 4 <= e;
    if (!kPerturb) {
      if (full) {
        *reinterpret_cast<uint2 *>(dst + g4) = *reinterpret_cast<const uint2 *>(src + g4);
      } else {
        for (int k = 0; k < 4; ++k)
          if (g4 + k >= b && g4 + k < e) dst[g4 + k] = src[g4 + k];
      }
      continue;
    }
    float th[4];
    if (full) {
      unpack4(*reinterpret_cast<const uint2 *>(backup + g4), th);
    } else {
      for (int k = 0; k < 4; ++k) th[k] = (g4 + k >= b && g4 + k < e) ? bf16_to_f32(backup[g4 + k]) : 0.0f;
    }
    uint32_t x[4];
    philox4x32_10_rk((uint32_t)(g4 >> 2), (uint32_t)(g4 >> 34), 0u, COPES_TAG_NOISE, a.rk, x);
    float xn[4], r[4], v[4], vp[4];
    normal_parts4_x2(x, a.coeffs.central2, a.coeffs.tail, xn, r);  // r = s sigma R(L)
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      v[k] = __fmaf_rn(r[k], xn[k], th[k]);
      vp[k] = __fmaf_rn(-r[k], xn[k], th[k]);
    }
    if (full) {
      *reinterpret_cast<uint2 *>(w + g4) = pack4(v);
      if (OP == kBackupPerturbPair) *reinterpret_cast<uint2 *>(pw + (g4 - a.partner_base)) = pack4(vp);
    } else {
      for (int k = 0; k < 4; ++k)
        if (g4 + k >= b && g4 + k < e) {
          w[g4 + k] = to_bf16_bits(v[k]);
          if (OP == kBackupPerturbPair) pw[g4 + k - a.partner_base] = to_bf16_bits(vp[k]);
        }
    }
  }
}

// The update: all P noise vectors regenerated per group in registers (noise_sum_groups,
// the tile update's loop), the backup read only after the noise loop, the new context
// written to both copies.  Same launch shape as the tile update: G groups per thread,
// 4 resident blocks per SM.
template <int G, bool HI0>
__device__ __forceinline__ void backup_update_tile(const UpdateArgs &a, uint16_t *backup, const float *s_w,
                                                   const uint32_t (*s_rk)[20], const uint32_t (*s_fk)[20],
                                                   uint64_t b, uint64_t e) {
  uint16_t *w = static_cast<uint16_t *>(a.w);
  for (uint64_t base = (b & ~3ull) + 4ull * threadIdx.x; base < e; base += 4ull * kThreads * G) {
    float acc[G][4];
    noise_sum_groups<G, HI0>(base, a.n_noise, s_w, s_rk, s_fk, acc);
#pragma unroll
    for (int i = 0; i < G; ++i) {
      const uint64_t g4 = base + 4ull * kThreads * i;
      if (g4 >= e) continue;
      if (g4 >= b && g4 + 4 <= e) {
        float th[4], v[4];
        unpack4(*reinterpret_cast<const uint2 *>(backup + g4), th);
#pragma unroll
        for (int k = 0; k < 4; ++k) v[k] = __fmaf_rn(a.coef, acc[i][k], th[k]);
        const uint2 p = pack4(v);
        *reinterpret_cast<uint2 *>(w + g4) = p;
        *reinterpret_cast<uint2 *>(backup + g4) = p;
      } else {
        for (int k = 0; k < 4; ++k) {
          const uint64_t g = g4 + k;
          if (g < b || g >= e) continue;
          const uint16_t h = to_bf16_bits(__fmaf_rn(a.coef, acc[i][k], bf16_to_f32(backup[g])));
          w[g] = h;
          backup[g] = h;
        }
      }
    }
  }
}

constexpr int kBackupUpdateGroups = 2;
constexpr int kBackupUpdateBlocksPerSM = 4;

__global__ void __launch_bounds__(kThreads, kBackupUpdateBlocksPerSM)
    backup_update_kernel(const __grid_constant__ UpdateArgs a, uint16_t *backup) {
  __shared__ float s_w[COPES_MAX_NOISE];
  __shared__ __align__(16) uint32_t s_rk[COPES_MAX_NOISE][20];
  __shared__ __align__(16) uint32_t s_fk[COPES_MAX_NOISE][20];
  noise_weights_to_smem(a, s_w, s_rk, s_fk);
  uint64_t b, e;
  if (!backup_tile(a.tiles, blockIdx.x, a.n_alloc, b, e)) return;
  if ((e >> 34) == 0) backup_update_tile<kBackupUpdateGroups, true>(a, backup, s_w, s_rk, s_fk, b, e);
  else backup_update_tile<kBackupUpdateGroups, false>(a, backup, s_w, s_rk, s_fk, b, e);
}

cudaError_t launch_backup_elementwise(int op, const ElemArgs &a, uint16_t *backup, cudaStream_t s) {
  if (a.n_tiles == 0) return cudaSuccess;
  const unsigned grid = (unsigned)a.n_tiles;
  switch (op) {
    case kBackupSave: backup_elem_kernel<kBackupSave><<<grid, kThreads, 0, s>>>(a, backup); break;
    case kBackupPerturb: backup_elem_kernel<kBackupPerturb><<<grid, kThreads, 0, s>>>(a, backup); break;
    case kBackupPerturbPair: backup_elem_kernel<kBackupPerturbPair><<<grid, kThreads, 0, s>>>(a, backup); break;
    default: backup_elem_kernel<kBackupRestore><<<grid, kThreads, 0, s>>>(a, backup); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_backup_update(const UpdateArgs &a, uint16_t *backup, cudaStream_t s) {
  if (a.n_tiles == 0) return cudaSuccess;
  backup_update_kernel<<<(unsigned)a.n_tiles, kThreads, 0, s>>>(a, backup);
  return cudaGetLastError();
}

unsigned read_and_clear_backup_errors() {
  unsigned v = 0, zero = 0;
  cudaMemcpyFromSymbol(&v, g_backup_error, sizeof(v));
  if (v) cudaMemcpyToSymbol(g_backup_error, &zero, sizeof(zero));
  return v;
}

}  // namespace copes
