/*
 * copes.h -- C ABI of the GB300 CoPES evolution-strategy core (libcopes.so).
 *
 * CoPES (Cooperative Parameter-subspace Evolution Strategy) perturbs one parameter
 * subspace S_k at a time while every other parameter keeps the shared context value
 * (Sec. 3.2, Eq. 8), standardises the population's scalar rewards (Eq. 5, Eq. 12), and
 * applies the reward-weighted update theta += c * sum_i f_i s_i eps_i (Eq. 6, Eq. 13),
 * regenerating every eps_i from its seed instead of storing it (Sec. 3.3 "Seed Replay,
 * Chunked Processing, and Weight Backup", Supp. A.8).
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Parameters live in ONE global index space.  Tensor t starts at offset off_t, with
 *    off_0 = 0 and off_{t+1} = off_t + numel_t rounded up to a multiple of 64
 *    (copes_layout).  The caller allocates two flat device buffers over that space: the
 *    working weights w (bf16 or fp32; what the model reads) and the fp32 master theta.
 *  - Noise: eps_seed[g] is a standard normal that depends only on (seed, g).  It is
 *    Phi^-1(u) of the odd-lattice uniform u = ((x & 0x7FFFFE) | 1) * 2^-23, where x is word
 *    (g & 3) of Philox4x32-10 (Salmon et al., SC'11) at counter (lo32(g >> 2),
 *    hi32(g >> 2), 0, 0) under key (lo32(seed), hi32(seed)).
 *  - Ownership: the caller owns every device buffer (weights, masters, rewards,
 *    fitness, subspace tables and lists, workspaces).  The library never allocates
 *    device memory.  Host arrays passed in are read during the call only.
 *  - Asynchrony: every call enqueues work on the caller's stream and returns; none
 *    synchronises unless its comment says so.  A stream of 0 is the legacy default
 *    stream.
 *  - Errors: calls return COPES_OK (0) or a negative COPES_ERR_* code and leave a
 *    thread-local message for copes_last_error().  Argument checks happen before any
 *    launch, so a failed call enqueues nothing.  Kernels never trap: a device-side
 *    range check that fails skips the access and raises a device error word, which
 *    copes_check() reports as COPES_ERR_DEVICE_CHECK.
 *  - Alignment: w and master must be 16-byte aligned (torch / cudaMalloc allocations
 *    are).  Subspace boundaries may fall anywhere; partial 4-element groups at the
 *    edges are handled element by element.
 */
#ifndef COPES_H
#define COPES_H

#include <stddef.h>
#include <stdint.h>

#ifndef __CUDA_RUNTIME_API_H__
typedef struct CUstream_st *cudaStream_t;
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------------- status codes */
enum {
  COPES_OK = 0,
  COPES_ERR_INVALID_ARG = -1,  /* null pointer, bad enum, inconsistent sizes */
  COPES_ERR_ALIGNMENT = -2,    /* w / master / list not aligned as documented */
  COPES_ERR_SIZE = -3,         /* a size outside the supported maximum */
  COPES_ERR_WORKSPACE = -4,    /* caller workspace or output capacity too small */
  COPES_ERR_CUDA = -5,         /* a CUDA runtime call failed (message has the text) */
  COPES_ERR_DEVICE_CHECK = -6, /* a kernel's own range check failed (see copes_check) */
  COPES_ERR_UNSUPPORTED = -7   /* a mode this library does not implement */
};

enum { COPES_BF16 = 0, COPES_FP32 = 1 };

/* Stream tags: independent Philox streams under the same seed. */
enum { COPES_TAG_NOISE = 0, COPES_TAG_INIT = 1, COPES_TAG_PARTITION = 2, COPES_TAG_SEED = 3,
       COPES_TAG_CHUNK = 4 };

/* Limits of this library version. */
enum {
  COPES_MAX_MEMBERS = 256,    /* population N per update call */
  COPES_MAX_NOISE = 256,      /* distinct noise vectors P per update call */
  COPES_MAX_K = 64,           /* subspaces per partition (hash mode) */
  COPES_TILE_MAX = 1 << 20    /* elements per subspace tile */
};

/* ------------------------------------------------------------------------- data types */

/* The flat parameter arena.
 * w2 (optional, NULL for none) is a second working-weight buffer of the same dtype and
 * size, for evaluating the two members of an antithetic pair on two copies of the model:
 * copes_perturb_pair with partner = w2, partner_base = 0, partner_len = n_alloc writes
 * member 2j's weights to w and member 2j+1's to w2 in one pass.  w3 and w4 (optional,
 * set together and only with w2) make four copies, on which copes_perturb_two_pairs
 * writes the four members of two antithetic pairs in one pass.  Restore, commit, the
 * fused update's commit and init write the context to every copy, so outside the live
 * subspace all of them always hold the context.  Perturbs write only the copies their
 * call names. */
typedef struct {
  void *w;          /* device: working weights, n_alloc elements of dtype              */
  float *master;    /* device: fp32 master theta, n_alloc elements                     */
  uint64_t n_alloc; /* elements in each buffer; every subspace index must be < n_alloc */
  int dtype;        /* COPES_BF16 or COPES_FP32 (the dtype of w)                       */
  void *w2;         /* device, optional: second working buffer (16-byte aligned), or NULL */
  void *w3;         /* device, optional: third working buffer (16-byte aligned), or NULL  */
  void *w4;         /* device, optional: fourth working buffer (16-byte aligned), or NULL */
} copes_params;
/* w, master, w2, w3 and w4 must be pairwise disjoint byte ranges (n_alloc elements
 * each): the kernels read the master while they write the working buffers.  Every call
 * that takes copes_params checks this, and that w3 and w4 come together and only with
 * w2, and returns COPES_ERR_INVALID_ARG otherwise.  A caller that zero-initialises the
 * struct and sets the first five fields gets one or two copies, as before w3 and w4. */

/* A subspace S (Eq. 7 / Eq. 8: the support of P_k).
 *  TILES:       a device array of n_tiles [begin, end) pairs of uint64 global indices
 *               (tiles[2i], tiles[2i+1]), each of at most COPES_TILE_MAX elements,
 *               pairwise disjoint.  Built by copes_subspace_build (range modes) or
 *               copes_tiles_from_ranges.
 *  INDICES:     a device array of n_index int64 global indices, strictly increasing (the
 *               gather form used for hash partitions).  The array must be 16-byte aligned.
 *  HASH_REPLAY: subspace k of the HASH partition (K, seed), with membership recomputed
 *               from the partition seed inside every kernel instead of read from a list
 *               (Supp. A.8 "Partition Replay"), or read from its optional membership
 *               mask.  Same members as the INDICES list that copes_hash_fill writes for
 *               (K, seed, k).  Filled by copes_hash_replay_subspace; `replay` is a device
 *               tensor table it writes. */
enum { COPES_SUBSPACE_TILES = 0, COPES_SUBSPACE_INDICES = 1, COPES_SUBSPACE_HASH_REPLAY = 2 };
typedef struct {
  int kind;
  const uint64_t *tiles;   /* TILES: device [2 * n_tiles]                                */
  uint64_t n_tiles;
  const int64_t *index;    /* INDICES: device [n_index]                                  */
  uint64_t n_index;
  const void *replay;      /* HASH_REPLAY: device tensor table (copes_hash_replay_subspace) */
  uint64_t n_replay_tiles; /* HASH_REPLAY: 16,384-element hash tiles the table covers     */
  int n_replay_tensors;    /* HASH_REPLAY: entries of the table                           */
  int K;                   /* HASH_REPLAY: subspaces of the partition, 1 <= K <= COPES_MAX_K */
  int k;                   /* HASH_REPLAY: this subspace, 0 <= k < K                      */
  uint64_t seed;           /* HASH_REPLAY: the partition seed                             */
  float *gathered;         /* INDICES, optional: device fp32 [n_index], the subspace's master
                              values in list order (see copes_gather_master); NULL: none */
  uint32_t *replay_mask;   /* HASH_REPLAY, optional: device membership bits filled by
                              copes_hash_replay_mask; NULL: membership is hashed */
} copes_subspace;

/* Parameter layout: the model's tensors in order. */
typedef struct {
  int n_tensors;
  const uint64_t *numel;     /* host [n_tensors]                                 */
  const uint32_t *tensor_id; /* host [n_tensors], or NULL for id = position      */
} copes_layout_desc;

/* Partition modes for copes_subspace_build. */
enum {
  COPES_PART_CONTIGUOUS = 0,    /* K consecutive slices of the parameters in layout order */
  COPES_PART_TENSOR_GROUPS = 1, /* union of the tensors with group id k                   */
  COPES_PART_HASH = 2,          /* per-element hash of (tensor id, element) -> index lists */
  COPES_PART_RANDOM_CHUNKS = 3  /* equal-size random partition of fixed-size chunks       */
};
typedef struct {
  int mode;
  int K;                   /* number of subspaces                                   */
  uint64_t seed;           /* HASH / RANDOM_CHUNKS: the partition seed             */
  uint64_t chunk;          /* RANDOM_CHUNKS: chunk size in global indices (>= 64, a
                              multiple of 64)                                         */
  const int32_t *group_of; /* TENSOR_GROUPS: host [n_tensors] group id per tensor  */
} copes_partition_spec;

/* Shaping modes for copes_shape_fitness. */
enum {
  COPES_SHAPE_NONE = 0,
  COPES_SHAPE_ZSCORE = 1,         /* Eq. 5 / Eq. 12: population z-score over all N      */
  COPES_SHAPE_ZSCORE_GROUPED = 2, /* Sec. 4.4: z-score within each group (subspace)    */
  COPES_SHAPE_CENTERED_RANK = 3   /* average ranks of ties, rank / (N - 1) - 1/2        */
};

enum { COPES_ONE_SIDED = 0, COPES_ANTITHETIC = 1 };
enum { COPES_COEF_PAPER = 0, COPES_COEF_OPENAI = 1 };

/* -------------------------------------------------------------------- host utilities */

/* Version string of the library (static storage).  0.2 added copes_params.w3 / w4 and
 * copes_perturb_two_pairs: callers built against 0.1's copes_params must be rebuilt. */
const char *copes_version(void);

/* Copies the calling thread's last error message into buf (NUL-terminated, truncated to
 * len) and returns the number of characters the full message has. */
int copes_last_error(char *buf, size_t len);

/* Synchronises `stream`, then reports and clears the device error words.  Returns
 * COPES_OK, COPES_ERR_DEVICE_CHECK (a kernel skipped an out-of-range access since the
 * last check) or COPES_ERR_CUDA (an asynchronous CUDA error surfaced). */
int copes_check(cudaStream_t stream);

/* Global offsets of a layout: offsets[0..n_tensors], offsets[n_tensors] = padded total.
 * offsets is a host array of n_tensors + 1 entries. */
int copes_layout(const copes_layout_desc *layout, uint64_t *offsets);

/* Eq. 11: sigma_k = sigma * sqrt(d / d_k) if dimension_aware, else sigma. */
double copes_sigma_eff(double sigma, double d, double d_k, int dimension_aware);

/* Step coefficient c of theta += c * sum_i s_i f_i eps_i:
 *   COPES_COEF_PAPER  (Eq. 6, Eq. 13): alpha / n_members
 *   COPES_COEF_OPENAI (theta += alpha / (N sigma) sum f eps): alpha / (n_members sigma_eff) */
double copes_step_coef(double alpha, int n_members, double sigma_eff, int convention);

/* Member table: ANTITHETIC maps member 2j -> (noise j, +1) and 2j+1 -> (noise j, -1);
 * ONE_SIDED maps member i -> (noise i, +1).  Host arrays of n_members entries.  Returns
 * the number of distinct noise vectors P (> 0) or a negative error code. */
int copes_member_table(int n_members, int pairing, int32_t *noise_id, int8_t *sign);

/* Seed of noise vector j of subspace k at iteration `iter`: the first two Philox words
 * (x0 | x1 << 32) at counter (j, k, iter, COPES_TAG_SEED) under key = base_seed. */
uint64_t copes_member_seed(uint64_t base_seed, uint32_t iter, uint32_t k, uint32_t j);

/* ------------------------------------------------------------------ subspace build
 * copes_subspace_build (Eq. 7; Algorithm 1 "sample a partition"; Supp. A.8 partition
 * replay) constructs subspace k of a K-way partition of the layout's parameters.
 *
 * Range modes (CONTIGUOUS, TENSOR_GROUPS, RANDOM_CHUNKS) produce a TILES subspace:
 *   call with tiles == NULL to get the tile count in *count (no device work for
 *   CONTIGUOUS / TENSOR_GROUPS), then again with a device buffer of 2 * count uint64;
 *   the tiles are written with an asynchronous copy on `stream` and *count is the number
 *   written.  tile_size (1 .. COPES_TILE_MAX) bounds the elements per tile.
 *   RANDOM_CHUNKS needs the chunk map: pass chunk_map (a device array of
 *   ceil(padded_total / chunk) uint32) built by copes_random_chunk_map; the call
 *   copies it to the host and SYNCHRONISES `stream`.
 * HASH mode produces an INDICES subspace; use copes_hash_count / copes_hash_fill.
 *
 * Contiguous slices cut the non-padding parameters, in layout order, at
 * floor(n k / K); groups take the union of the tensors with group id k; random chunks
 * take the chunks the map assigns to k, intersected with the tensors. */
int copes_subspace_build(const copes_layout_desc *layout, const copes_partition_spec *spec,
                         int k, uint64_t tile_size, const uint32_t *chunk_map,
                         uint64_t *tiles, uint64_t capacity, uint64_t *count,
                         cudaStream_t stream);

/* Tiles of an arbitrary list of host ranges [begin[i], end[i]) (adjacent ranges are
 * merged; ranges must not overlap).  Same two-call protocol and asynchronous copy as
 * copes_subspace_build. */
int copes_tiles_from_ranges(const uint64_t *begin, const uint64_t *end, int n_ranges,
                            uint64_t tile_size, uint64_t *tiles, uint64_t capacity,
                            uint64_t *count, cudaStream_t stream);

/* RANDOM_CHUNKS map: chunk c (global indices [c chunk, (c+1) chunk)) gets key = word 0
 * of Philox(seed; c, 0, COPES_TAG_CHUNK); chunks ranked by (key, c) go to subspace
 * floor(rank K / n_chunks), so subspace sizes differ by at most one chunk.  Writes
 * n_chunks uint32 to the device array map.  n_chunks <= 2^20.  workspace: device memory
 * of copes_random_chunk_map_workspace_bytes(n_chunks) bytes (8 per chunk, the count
 * rounded up to a power of two of at least 4,096), 16-byte aligned; the ranks come from
 * a sort of the chunks' keys there.  Asynchronous. */
size_t copes_random_chunk_map_workspace_bytes(uint64_t n_chunks);
int copes_random_chunk_map(uint64_t n_chunks, int K, uint64_t seed, uint32_t *map,
                           void *workspace, size_t workspace_bytes, cudaStream_t stream);

/* HASH partition, phase 1: element e of tensor tid goes to subspace
 * floor(x K / 2^32) with x = word (e & 3) of Philox(seed; e >> 2, tid, COPES_TAG_PARTITION).
 * Counts the members of every subspace into counts[K] (host) and SYNCHRONISES `stream`.
 * workspace: device memory of copes_hash_workspace_bytes() bytes (16-byte aligned). */
size_t copes_hash_workspace_bytes(const copes_layout_desc *layout, int K);
int copes_hash_count(const copes_layout_desc *layout, int K, uint64_t seed, void *workspace,
                     size_t workspace_bytes, uint64_t *counts, cudaStream_t stream);

/* HASH partition, phase 2: writes the sorted global-index list of every subspace k into
 * lists[k] (host array of K device pointers; lists[k] holds counts[k] int64 from phase
 * 1).  Requires the workspace filled by copes_hash_count with the same arguments.
 * Asynchronous. */
int copes_hash_fill(const copes_layout_desc *layout, int K, uint64_t seed, void *workspace,
                    size_t workspace_bytes, int64_t *const *lists, cudaStream_t stream);

/* Hash partition for callers that cannot allocate device memory -- for instance an ES
 * trainer sharing the GPU with a rollout engine that reserved nearly all free HBM for its
 * KV cache, or code inside a framework that owns the memory pool and forbids cudaMalloc.
 * (The paper has no counterpart: this is a deployment variant of copes_hash_count +
 * copes_hash_fill.)  Same partition and same output as those two calls, but the scratch
 * is a fixed 8 MiB array inside the library, held by every GPU that loads it until the
 * process exits; nothing is allocated on the device or the host.
 *  - lists == NULL: counts every subspace into counts[K] (host) and SYNCHRONISES stream.
 *  - otherwise also writes the sorted lists: lists[k] (device, capacity[k] int64, host
 *    arrays of K) must hold counts[k] entries, else COPES_ERR_WORKSPACE and no list is
 *    written; the fill is asynchronous on stream.
 * A layout whose scratch exceeds 8 MiB (about 12 K bytes per 16,384-element tile) is
 * rejected with COPES_ERR_SIZE.  The first call on a device looks up the array's device
 * address with that device current; make that first call before any stream capture.
 * Every call reuses the same array, so calls whose GPU work overlaps race: serialise them. */
int copes_hash_partition_static(const copes_layout_desc *layout, int K, uint64_t seed,
                                int64_t *const *lists, const uint64_t *capacity,
                                uint64_t *counts, cudaStream_t stream);

/* Gathered master of an INDICES subspace (no counterpart in the paper: a memory-layout
 * option for scattered subspaces).  With S->gathered set, perturb, restore, commit, init
 * and update over S read theta from gathered[p] for the p-th index (and the update and
 * init write it there) instead of master[index[p]]; master is not touched.  The results
 * are those of the master path, bit for bit, while the master reads become contiguous
 * (4 bytes per member instead of a 32-byte sector of master each).
 *  copes_gather_master:  gathered[p] = master[index[p]]   (before the subspace's visits)
 *  copes_scatter_master: master[index[p]] = gathered[p]   (to publish theta back)
 * Both need S->kind == INDICES and S->gathered (16-byte aligned); asynchronous. */
int copes_gather_master(const copes_params *p, const copes_subspace *S, cudaStream_t stream);
int copes_scatter_master(const copes_params *p, const copes_subspace *S, cudaStream_t stream);

/* HASH partition by replay (Supp. A.8 "Partition Replay": the partition is kept as its
 * seed and replayed, not stored as a parameter-level assignment).  Writes the layout's
 * replay table (copes_hash_replay_bytes() bytes: 32 per non-empty tensor, rounded up to
 * 16, plus 4 per 16,384-element tile, rounded up to 16) into the device buffer `table`
 * (16-byte aligned, caller-owned; it must outlive every call that uses *out) with
 * asynchronous copies on `stream`, and fills *out as the HASH_REPLAY subspace k of the
 * partition (K, seed).  No list is built: perturb, restore, commit and update over *out
 * recompute, per 16,384-element tile, each element's bucket floor(x K / 2^32) (x as in
 * copes_hash_count), gather the members of subspace k in shared memory and process them.
 * Results are identical to those over the INDICES list of (K, seed, k).  The table does
 * not depend on K, seed or k, so the K subspaces of one partition may share one table. */
size_t copes_hash_replay_bytes(const copes_layout_desc *layout);

int copes_hash_replay_subspace(const copes_layout_desc *layout, int K, uint64_t seed, int k,
                               void *table, size_t table_bytes, cudaStream_t stream,
                               copes_subspace *out);

/* Membership mask of a HASH_REPLAY subspace (a cache of its replay, no counterpart in the
 * paper): one bit per element, 2,048 bytes per 16,384-element hash tile
 * (S->n_replay_tiles * 2048 bytes, 16-byte aligned, in S->replay_mask, caller-owned).
 * Hashes every element once and writes the bits of subspace S->k; afterwards the ES steps
 * over S read the bits instead of hashing.  Meant to be built at the start of a visit and
 * reused by its perturbs, restore and update; rebuild it when S's partition (K, k, seed)
 * or table changes.  Asynchronous. */
int copes_hash_replay_mask(const copes_params *p, const copes_subspace *S, cudaStream_t stream);

/* ------------------------------------------------------------------------- ES steps */

/* Perturb (Eq. 8, Algorithm 1 "set theta_{k,i}"): for every g in S,
 *   w[g] = round(fma(signed_sigma, eps_seed[g], theta[g]))   (fp32 fma, then RNE to bf16)
 * Every element outside S is left untouched.  Reads theta (never w), so the call is
 * idempotent and no restore is needed between members.  signed_sigma = s * sigma_k
 * carries the antithetic sign. */
int copes_perturb(const copes_params *p, const copes_subspace *S, uint64_t seed,
                  float signed_sigma, cudaStream_t stream);

/* Antithetic pair perturb (Eq. 8 for both members of one noise vector, no counterpart in
 * the paper's implementation): one pass over S computes, for every g in S,
 *   w[g]                          = round(fma( signed_sigma, eps_seed[g], theta[g]))
 *   partner[g - partner_base]     = round(fma(-signed_sigma, eps_seed[g], theta[g]))
 * i.e. w exactly as copes_perturb(signed_sigma) writes it, and the partner member's
 * weights exactly as copes_perturb(-signed_sigma) would write them, from one generation
 * of the noise.  partner: caller-owned device buffer of the working dtype (2 B per element
 * for bf16, 4 B for fp32), 16-byte aligned, holding global indices
 * [partner_base, partner_base + partner_len) at offsets 0 .. partner_len - 1; partner_base
 * is a multiple of 4, the range lies inside the arena and the buffer overlaps neither w
 * nor the master (COPES_ERR_ALIGNMENT / COPES_ERR_SIZE / COPES_ERR_INVALID_ARG otherwise).  It may be the
 * arena's second working buffer w2.  An element of S outside that range is skipped and reported
 * by copes_check (bit 16).  Entries of the buffer outside S are untouched. */
int copes_perturb_pair(const copes_params *p, const copes_subspace *S, uint64_t seed,
                       float signed_sigma, void *partner, uint64_t partner_base,
                       uint64_t partner_len, cudaStream_t stream);

/* The partner member's perturb: w[g] = partner[g - partner_base] for g in S, a copy of
 * the values copes_perturb_pair wrote.  Equal, bit for bit, to copes_perturb with the
 * partner's signed sigma as long as theta is unchanged since that copes_perturb_pair.
 * Reads neither theta nor the noise.  Buffer rules as for copes_perturb_pair. */
int copes_perturb_partner(const copes_params *p, const copes_subspace *S, const void *partner,
                          uint64_t partner_base, uint64_t partner_len, cudaStream_t stream);

/* Two antithetic pairs in one pass (Eq. 8 for the four members of two noise vectors; no
 * counterpart in the paper's implementation).  With four working copies (p->w2, p->w3
 * and p->w4 set), for every g in S:
 *   w[g]  = round(fma( signed_sigma, eps_seed_a[g], theta[g]))
 *   w2[g] = round(fma(-signed_sigma, eps_seed_a[g], theta[g]))
 *   w3[g] = round(fma( signed_sigma, eps_seed_b[g], theta[g]))
 *   w4[g] = round(fma(-signed_sigma, eps_seed_b[g], theta[g]))
 * each exactly what copes_perturb writes with that seed and signed sigma, from one read
 * of theta.  Elements outside S are untouched.  TILES subspaces only
 * (COPES_ERR_UNSUPPORTED otherwise); without four copies COPES_ERR_INVALID_ARG. */
int copes_perturb_two_pairs(const copes_params *p, const copes_subspace *S, uint64_t seed_a,
                            uint64_t seed_b, float signed_sigma, cudaStream_t stream);

/* Restore (Sec. 3.3, Supp. A.8 "CPU Weight Backup", here an on-device fp32 master):
 *   w[g] = round(theta[g]) for g in S, bit-exact; outside S untouched.  Every further
 * working copy (w2, w3, w4) that p sets gets the same value. */
int copes_restore(const copes_params *p, const copes_subspace *S, cudaStream_t stream);

/* Context commit (Sec. 3.2 shared context after Eq. 13): w[g] = round(theta[g]) for
 * g in S (and in every further working copy p sets).  Same arithmetic as copes_restore,
 * called after copes_update. */
int copes_context_commit(const copes_params *p, const copes_subspace *S, cudaStream_t stream);

/* Fitness shaping (Eq. 5, Eq. 12, Sec. 4.4): f = shape(r) over n rewards (device fp32),
 * statistics in fp64.  group (device int32 [n]) is read only by ZSCORE_GROUPED.  A pool
 * whose rewards are all equal gets f = 0.  n <= COPES_MAX_MEMBERS. */
int copes_shape_fitness(const float *rewards, int n, const int32_t *group, int mode,
                        float *fitness, cudaStream_t stream);

/* Update (Eq. 6, Eq. 13, Algorithm 1): for every g in S,
 *   theta[g] = fma(coef, acc, theta[g]),  acc = sum_j w_j eps_{seeds[j]}[g]  (fp32),
 *   w_j = sum over members i with noise_id[i] == j of sign[i] * fitness[i].
 * All n_noise noise vectors are regenerated in registers in one pass; nothing is
 * stored.  noise_id, sign (host, n_members) and seeds (host, n_noise) are read during
 * the call; fitness is device fp32 [n_members].  fuse_commit != 0 also writes
 * w[g] = round(theta[g]) (the context commit, to every working copy p sets) in the
 * same pass. */
int copes_update(const copes_params *p, const copes_subspace *S, int n_members,
                 const int32_t *noise_id, const int8_t *sign, const float *fitness,
                 int n_noise, const uint64_t *seeds, float coef, int fuse_commit,
                 cudaStream_t stream);

/* Synthetic initialisation (input preparation, not part of the method): for g in S,
 *   theta[g] = mean + scale * eps_seed^(INIT)[g],  w[g] = round(theta[g])  (and every
 * further working copy). */
int copes_init_normal(const copes_params *p, const copes_subspace *S, uint64_t seed,
                      float mean, float scale, cudaStream_t stream);

/* ----------------------------------------------------------- CPU weight backup mode */

/* CPU weight backup (Supp. A.8 "CPU Weight Backup"): for a GPU on which an fp32 master
 * does not fit, the working weights stay bf16 in HBM and the pre-perturbation weights
 * (the shared context) are kept as a bf16 copy in pinned host memory, which the kernels
 * read and write directly (on GB300 across NVLink-C2C).  Perturbations are computed from
 * the backup, never from the live weights, so every member is evaluated from the same
 * pre-update model and perturb stays idempotent; restore copies the backup back, with no
 * subtraction of replayed noise.
 *  w:       device bf16 [n_alloc], the weights the model reads;
 *  backup:  host bf16 [n_alloc] in page-locked memory (cudaHostAlloc / cudaHostRegister,
 *           or torch's pin_memory()); any other pointer gives COPES_ERR_INVALID_ARG.
 * Only TILES subspaces are supported (COPES_ERR_UNSUPPORTED otherwise).  Both buffers are
 * indexed by the global index g, like w and master in copes_params. */
typedef struct {
  void *w;           /* device bf16 [n_alloc]                 */
  uint16_t *backup;  /* pinned host bf16 [n_alloc]            */
  uint64_t n_alloc;
} copes_backup_params;

/* backup[g] = w[g] for g in S (the context is saved before the members are evaluated). */
int copes_backup_save(const copes_backup_params *p, const copes_subspace *S, cudaStream_t stream);

/* Perturb from the backup (Eq. 8): w[g] = round(fma(signed_sigma, eps_seed[g], backup[g])). */
int copes_backup_perturb(const copes_backup_params *p, const copes_subspace *S, uint64_t seed,
                         float signed_sigma, cudaStream_t stream);

/* Antithetic pair perturb from the backup: w as copes_backup_perturb(signed_sigma) and
 * partner[g - partner_base] = round(fma(-signed_sigma, eps_seed[g], backup[g])), the
 * partner member's weights, from one read of the backup over the host link.  The partner
 * buffer is device memory, bf16, with the rules of copes_perturb_pair (its device range
 * check reports bit 16 in copes_check). */
int copes_backup_perturb_pair(const copes_backup_params *p, const copes_subspace *S, uint64_t seed,
                              float signed_sigma, void *partner, uint64_t partner_base,
                              uint64_t partner_len, cudaStream_t stream);

/* The partner member's perturb: w[g] = partner[g - partner_base] for g in S (device to
 * device, no host-link traffic). */
int copes_backup_perturb_partner(const copes_backup_params *p, const copes_subspace *S,
                                 const void *partner, uint64_t partner_base, uint64_t partner_len,
                                 cudaStream_t stream);

/* Restore (Supp. A.8): w[g] = backup[g], bit-exact. */
int copes_backup_restore(const copes_backup_params *p, const copes_subspace *S, cudaStream_t stream);

/* Update from the backup (Eq. 6, Eq. 13), with the arguments of copes_update:
 *   t = fma(coef, acc, backup[g]) in fp32,  w[g] = backup[g] = round(t),
 * so the new context is both published to the model and saved as the next backup. */
int copes_backup_update(const copes_backup_params *p, const copes_subspace *S, int n_members,
                        const int32_t *noise_id, const int8_t *sign, const float *fitness,
                        int n_noise, const uint64_t *seeds, float coef, cudaStream_t stream);

/* ------------------------------------------------------------------- debug exports */

/* Philox words for counters q0 .. q0+n-1 with (aux, tag): out is device uint32 [4n]. */
int copes_debug_philox(uint64_t seed, uint64_t q0, uint64_t n, uint32_t aux, uint32_t tag,
                       uint32_t *out, cudaStream_t stream);

/* eps_seed^(tag)[g] for g = g0 .. g0+n-1: out is device fp32 [n]. */
int copes_debug_normals(uint64_t seed, uint32_t tag, uint64_t g0, uint64_t n, float *out,
                        cudaStream_t stream);

/* The word -> normal transform alone: out[i] = normal(words[i]) (device arrays). */
int copes_debug_transform(const uint32_t *words, uint64_t n, float *out, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* COPES_H */
