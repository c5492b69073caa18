// Internal declarations shared by the host API and the kernel translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/copes.h"
#include "normal_coeffs.h"

namespace copes {

constexpr int kThreads = 256;       // threads per block of the elementwise kernels
constexpr int kIndexSegment = 8192; // indices per block in the gather kernels

// Philox4x32-10 constants (SC'11, Sec. 3): round multipliers and key (Weyl) increments.
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

// Philox4x32-10 on one counter: 10 rounds of (two 32x32->64 multiplies, XOR of the high
// halves with the other counter words and the round key, key bump).  Host and device.
__host__ __device__ __forceinline__ void philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2,
                                                       uint32_t c3, uint32_t k0, uint32_t k1,
                                                       uint32_t out[4]) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)kPhiloxM0 * c0;
    const uint64_t p1 = (uint64_t)kPhiloxM1 * c2;
    const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
    const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
    c1 = (uint32_t)p1;
    c3 = (uint32_t)p0;
    c0 = n0;
    c2 = n2;
    k0 += kPhiloxW0;
    k1 += kPhiloxW1;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

// Round keys of Philox4x32-10: rk[2r] = k0 + r W0, rk[2r+1] = k1 + r W1 (r = 0..9).
__host__ __device__ __forceinline__ void philox_round_keys(uint32_t k0, uint32_t k1, uint32_t rk[20]) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    rk[2 * r] = k0 + (uint32_t)r * kPhiloxW0;
    rk[2 * r + 1] = k1 + (uint32_t)r * kPhiloxW1;
  }
}

// The same generator with the key schedule precomputed: the per-round key additions
// are taken out of the hot loop (rk may live in the constant bank or shared memory).
template <typename RK>
__host__ __device__ __forceinline__ void philox4x32_10_rk(uint32_t c0, uint32_t c1, uint32_t c2,
                                                          uint32_t c3, const RK &rk,
                                                          uint32_t out[4]) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)kPhiloxM0 * c0;
    const uint64_t p1 = (uint64_t)kPhiloxM1 * c2;
    const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ rk[2 * r];
    const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ rk[2 * r + 1];
    c1 = (uint32_t)p1;
    c3 = (uint32_t)p0;
    c0 = n0;
    c2 = n2;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

// Philox4x32-10 at a counter (c0, 0, 0, tag) -- high word and aux zero -- with the work that
// does not depend on c0 taken out.  With c1 = c2 = 0, round 0's second product is 0 and
//   round 0: (c0, c1, c2, c3) <- (k0, 0, hi(M0 c0) ^ tag ^ k1, lo(M0 c0));
//   round 1: M0 * k0 is a function of the key alone, so
//            (c0, c1, c2, c3) <- (hi(M1 c2) ^ rk2, lo(M1 c2), hi(M0 k0) ^ lo(M0 c0) ^ rk3, lo(M0 k0));
//   round 2: its c3 = lo(M0 k0) enters only word 2, XORed with rk5.
// philox_folded_keys gathers those key-only terms with the remaining round keys:
//   u = {k1 ^ tag, rk2, hi(M0 k0) ^ rk3, lo(M0 k0) ^ rk5, rk4, rk6, rk7, ..., rk19, 0};
// philox4x32_10_folded then takes the counter's product M0 * c0 (which a caller computes
// once for every key) and runs one multiply in round 1 and two in each of rounds 2..9:
// 17 of the 20 32x32->64 multiplies, with the same output words as philox4x32_10.
__host__ __device__ __forceinline__ void philox_folded_keys(const uint32_t rk[20], uint32_t tag, uint32_t u[20]) {
  const uint64_t mk = (uint64_t)kPhiloxM0 * rk[0];
  u[0] = rk[1] ^ tag;
  u[1] = rk[2];
  u[2] = (uint32_t)(mk >> 32) ^ rk[3];
  u[3] = (uint32_t)mk ^ rk[5];
  u[4] = rk[4];
  for (int r = 3; r < 10; ++r) {
    u[5 + 2 * (r - 3)] = rk[2 * r];
    u[6 + 2 * (r - 3)] = rk[2 * r + 1];
  }
  u[19] = 0;
}

template <typename U>
__host__ __device__ __forceinline__ void philox4x32_10_folded(uint32_t m0_lo, uint32_t m0_hi, const U &u,
                                                              uint32_t out[4]) {
  uint32_t c2 = m0_hi ^ u[0];  // after round 0
  uint64_t p1 = (uint64_t)kPhiloxM1 * c2;
  uint32_t c0 = (uint32_t)(p1 >> 32) ^ u[1];  // after round 1
  uint32_t c1 = (uint32_t)p1;
  c2 = u[2] ^ m0_lo;
  uint64_t p0 = (uint64_t)kPhiloxM0 * c0;  // round 2
  p1 = (uint64_t)kPhiloxM1 * c2;
  c0 = (uint32_t)(p1 >> 32) ^ c1 ^ u[4];
  c2 = (uint32_t)(p0 >> 32) ^ u[3];
  c1 = (uint32_t)p1;
  uint32_t c3 = (uint32_t)p0;
#pragma unroll
  for (int r = 3; r < 10; ++r) {
    p0 = (uint64_t)kPhiloxM0 * c0;
    p1 = (uint64_t)kPhiloxM1 * c2;
    const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ u[5 + 2 * (r - 3)];
    const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ u[6 + 2 * (r - 3)];
    c1 = (uint32_t)p1;
    c3 = (uint32_t)p0;
    c0 = n0;
    c2 = n2;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

// Device error bits (set with atomicOr by a kernel that skipped an access).
enum : unsigned {
  kErrTileRange = 1u,   // a tile outside [0, n_alloc) or longer than COPES_TILE_MAX
  kErrIndexRange = 2u,  // a gather index outside [0, n_alloc)
  kErrPartition = 4u,   // a partition kernel met an inconsistent workspace
  kErrStageTimeout = 8u, // a bulk-copy wait ran past its iteration limit
  kErrPartnerRange = 16u // an element outside the partner buffer's range
};

// ---------------------------------------------------------------- launch arguments
// R's coefficients pre-multiplied by the perturbation scale (filled by the host).
struct ScaledCoeffs {
  unsigned long long central2[COPES_NORMAL_CENTRAL_DEGREE + 1];  // (c, c) pairs
  float central[COPES_NORMAL_CENTRAL_DEGREE + 1];
  float tail[COPES_NORMAL_TAIL_DEGREE + 1];
};

// The working copies beyond w (copes_params.w2, w3, w4): n = 0, 1 (w2) or 3 (w2, w3, w4).
struct WorkingCopies {
  void *p[3];
  int n;
};

struct ElemArgs {
  void *w;
  float *master;
  uint64_t n_alloc;
  const uint64_t *tiles;
  uint64_t n_tiles;
  const int64_t *index;
  uint64_t n_index;
  uint32_t seed_lo, seed_hi;
  uint32_t tag;
  float a;  // perturb: signed sigma; init: scale
  float b;  // init: mean
  ScaledCoeffs coeffs;  // a * R's coefficients (perturb, init)
  uint32_t rk[20];      // Philox round keys of (seed_lo, seed_hi)
  float *gathered;      // INDICES: theta in list order instead of master[index[p]] (or NULL)
  // kOpPerturbPair / kOpPartner: the antithetic partner's weights (working dtype), element
  // g at partner[g - partner_base] for partner_base <= g < partner_base + partner_len
  void *partner;
  uint64_t partner_base, partner_len;
  WorkingCopies copies;  // restore / commit / init write these as well as w
  // kOpPerturbTwoPairs: the second noise vector's round keys, and both vectors' folded keys
  // (philox_folded_keys, noise tag) for counters below 2^32
  uint32_t rk_b[20];
  uint32_t fk[20], fk_b[20];
};

// kOpGather / kOpScatter copy theta between master and the gathered copy (INDICES only).
// kOpPerturbPair writes w = rn(theta + a eps) and the partner member's rn(theta - a eps)
// to the partner buffer; kOpPartner copies the partner buffer into w.  kOpPerturbTwoPairs
// (TILES only, three further working copies) writes rn(theta + a eps) and
// rn(theta - a eps) for the first noise vector to w and copies[0], and for the second
// (keys rk_b) to copies[1] and copies[2].
enum ElemOp {
  kOpPerturb = 0,
  kOpRestore = 1,
  kOpInit = 2,
  kOpGather = 3,
  kOpScatter = 4,
  kOpPerturbPair = 5,
  kOpPartner = 6,
  kOpPerturbTwoPairs = 7
};

struct UpdateArgs {
  void *w;
  float *master;
  uint64_t n_alloc;
  const uint64_t *tiles;
  uint64_t n_tiles;
  const int64_t *index;
  uint64_t n_index;
  const float *fitness;
  float coef;
  int n_members;
  int n_noise;
  int fuse_commit;
  uint32_t seed_lo[COPES_MAX_NOISE];
  uint32_t seed_hi[COPES_MAX_NOISE];
  uint16_t noise_ptr[COPES_MAX_NOISE + 1];  // members of noise j: noise_member[ptr[j] .. ptr[j+1])
  uint16_t noise_member[COPES_MAX_MEMBERS];
  int8_t sign[COPES_MAX_MEMBERS];
  float *gathered;  // INDICES: theta in list order instead of master[index[p]] (or NULL)
  WorkingCopies copies;  // the fused commit writes these as well as w
};

// ------------------------------------------------------------------------ launchers
// Each returns the launch's cudaError_t (cudaSuccess when nothing was launched).
cudaError_t launch_elementwise(int op, int kind, int dtype, const ElemArgs &a, cudaStream_t s);
cudaError_t launch_update(int kind, int dtype, const UpdateArgs &a, cudaStream_t s,
                          int num_sms);
cudaError_t launch_shape(const float *r, int n, const int32_t *group, int mode, float *f,
                         cudaStream_t s);
cudaError_t launch_debug_philox(uint64_t seed, uint64_t q0, uint64_t n, uint32_t aux,
                                uint32_t tag, uint32_t *out, cudaStream_t s);
cudaError_t launch_debug_normals(uint64_t seed, uint32_t tag, uint64_t g0, uint64_t n,
                                 float *out, cudaStream_t s);
cudaError_t launch_debug_transform(const uint32_t *words, uint64_t n, float *out,
                                   cudaStream_t s);

// Hash partition.  The workspace begins with a table of HashTensor entries, then per
// hash tile a K-bucket histogram (uint32), then per hash tile K exclusive offsets
// (uint64), then K totals (unsigned long long).
constexpr uint64_t kHashTile = 16384;
struct HashTensor {
  uint64_t offset;      // global offset of the tensor
  uint64_t numel;
  uint64_t tile_begin;  // first hash tile of the tensor
  uint32_t tensor_id;
  uint32_t pad;
};
static_assert(sizeof(HashTensor) == 32, "the replay table is documented as 32 bytes per tensor");
cudaError_t launch_hash_hist(const HashTensor *tensors, int n_tensors, uint64_t n_htiles, int K,
                             uint64_t seed, uint32_t *hist, unsigned long long *totals,
                             cudaStream_t s);
cudaError_t launch_hash_scan(const uint32_t *hist, uint64_t n_htiles, int K, uint64_t *offsets,
                             cudaStream_t s);
cudaError_t launch_hash_scatter(const HashTensor *tensors, int n_tensors, uint64_t n_htiles,
                                int K, uint64_t seed, const uint64_t *offsets,
                                int64_t *const *lists, cudaStream_t s);
// A tile table's ranges as launch parameters: range r covers [begin[r], end[r]) and its
// tiles start at index first[r]; first[n_ranges] is the tile count.
constexpr int kTileRangesMax = 1000;
struct TileRanges {
  uint64_t begin[kTileRangesMax];
  uint64_t end[kTileRangesMax];
  uint64_t first[kTileRangesMax + 1];
  uint64_t tile_size;
  int n_ranges;
};
cudaError_t launch_tile_expand(const TileRanges &r, uint64_t *tiles, cudaStream_t s);
// keys: workspace of chunk_sort_size(n_chunks) uint64.
uint64_t chunk_sort_size(uint64_t n_chunks);
cudaError_t launch_random_chunk_map(uint64_t n_chunks, int K, uint64_t seed, uint32_t *map,
                                    uint64_t *keys, cudaStream_t s);

// Partition replay: subspace k of the hash partition (K, seed), recomputed per hash tile
// from the replay table: one HashTensor per non-empty tensor (layout order), then, from
// the next 16-byte boundary, the table entry (uint32) of every hash tile.
struct ReplayArgs {
  const HashTensor *table;
  const uint32_t *tile_tensor;  // table entry of each hash tile
  int n_tensors;
  uint64_t n_tiles;  // hash tiles of kHashTile elements covered by the table
  uint32_t seed_lo, seed_hi;
  int K, k;
  // bucket k is the word range [lo, lo + span] (32-bit unsigned): lo = ceil(k 2^32 / K),
  // span = ceil((k + 1) 2^32 / K) - lo - 1 (2^32 - 1 when K = 1)
  uint32_t lo, span;
  uint32_t rk[20];  // Philox round keys of the partition seed
  const uint32_t *mask;  // membership bits (copes_hash_replay_mask), or NULL: hash
};
cudaError_t launch_replay_elementwise(int op, int dtype, const ElemArgs &a, const ReplayArgs &r,
                                      cudaStream_t s);
cudaError_t launch_replay_update(int dtype, const UpdateArgs &a, const ReplayArgs &r,
                                 cudaStream_t s);
cudaError_t launch_replay_mask(const ReplayArgs &r, uint64_t n_alloc, uint32_t *mask, cudaStream_t s);

// CPU weight backup mode: `backup` is the device-accessible pointer of pinned host memory.
// kBackupPerturbPair: w = round(theta + a eps) and the antithetic partner's
// round(theta - a eps) into ElemArgs.partner, theta = the backup, read over the link once.
enum BackupOp { kBackupSave = 0, kBackupPerturb = 1, kBackupRestore = 2, kBackupPerturbPair = 3 };
cudaError_t launch_backup_elementwise(int op, const ElemArgs &a, uint16_t *backup, cudaStream_t s);
cudaError_t launch_backup_update(const UpdateArgs &a, uint16_t *backup, cudaStream_t s);

// Sets the calling thread's message reported by copes_last_error.
void set_last_error(const char *message);

// Device error words of each translation unit: read and clear (synchronous).
unsigned read_and_clear_es_errors();
unsigned read_and_clear_partition_errors();
unsigned read_and_clear_replay_errors();
unsigned read_and_clear_backup_errors();

}  // namespace copes
