// Host side of the C ABI: argument checks, subspace construction, member tables and the
// kernel launches.  Every public function validates everything it can before it
// enqueues anything, and reports failures through a status code plus a thread-local
// message.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <utility>
#include <vector>

#include "copes_internal.h"
#include "normal_coeffs.h"

using copes::ElemArgs;
using copes::UpdateArgs;

namespace {

thread_local std::string g_message;

int fail(int code, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_message = buf;
  return code;
}

int cuda_fail(cudaError_t e, const char *what) {
  return fail(COPES_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// True when the byte ranges [a, a + na) and [b, b + nb) overlap.
static bool overlaps(const void *a, uint64_t na, const void *b, uint64_t nb) {
  const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
  return a && b && na && nb && x < y + nb && y < x + na;
}

static uint64_t elem_size(int dtype) { return dtype == COPES_BF16 ? 2 : 4; }

int check_params(const copes_params *p, const char *who) {
  if (!p) return fail(COPES_ERR_INVALID_ARG, "%s: params is NULL", who);
  if (!p->w || !p->master) return fail(COPES_ERR_INVALID_ARG, "%s: w or master is NULL", who);
  if (p->dtype != COPES_BF16 && p->dtype != COPES_FP32)
    return fail(COPES_ERR_INVALID_ARG, "%s: dtype %d is neither COPES_BF16 nor COPES_FP32", who,
                p->dtype);
  if (!aligned(p->w, 16) || !aligned(p->master, 16))
    return fail(COPES_ERR_ALIGNMENT, "%s: w and master must be 16-byte aligned", who);
  if ((p->w3 == nullptr) != (p->w4 == nullptr))
    return fail(COPES_ERR_INVALID_ARG, "%s: w3 and w4 are set together", who);
  if (p->w3 && !p->w2) return fail(COPES_ERR_INVALID_ARG, "%s: w3 and w4 need w2", who);
  if (!aligned(p->w2, 16) || !aligned(p->w3, 16) || !aligned(p->w4, 16))
    return fail(COPES_ERR_ALIGNMENT, "%s: w2, w3 and w4 must be 16-byte aligned", who);
  if (p->n_alloc == 0) return fail(COPES_ERR_SIZE, "%s: n_alloc is 0", who);
  // the kernels read master while they write the working copies: all must be disjoint
  const uint64_t wbytes = p->n_alloc * elem_size(p->dtype), mbytes = p->n_alloc * 4;
  if (overlaps(p->w, wbytes, p->master, mbytes))
    return fail(COPES_ERR_INVALID_ARG, "%s: w and master overlap", who);
  const void *extra[3] = {p->w2, p->w3, p->w4};
  static const char *name[3] = {"w2", "w3", "w4"};
  for (int i = 0; i < 3; ++i) {
    if (!extra[i]) continue;
    if (extra[i] == p->w || extra[i] == (const void *)p->master)
      return fail(COPES_ERR_INVALID_ARG, "%s: %s must be a buffer of its own", who, name[i]);
    if (overlaps(extra[i], wbytes, p->w, wbytes) || overlaps(extra[i], wbytes, p->master, mbytes))
      return fail(COPES_ERR_INVALID_ARG, "%s: %s overlaps w or master", who, name[i]);
    for (int j = 0; j < i; ++j)
      if (extra[j] && (extra[j] == extra[i] || overlaps(extra[i], wbytes, extra[j], wbytes)))
        return fail(COPES_ERR_INVALID_ARG, "%s: %s overlaps %s", who, name[i], name[j]);
  }
  return COPES_OK;
}

// The working copies beyond w, in order: none, w2, or w2, w3, w4 (check_params enforces
// that w3 and w4 come together and only with w2).
copes::WorkingCopies working_copies(const copes_params *p) {
  copes::WorkingCopies c{};
  c.p[0] = p->w2;
  c.p[1] = p->w3;
  c.p[2] = p->w4;
  c.n = p->w4 ? 3 : (p->w2 ? 1 : 0);
  return c;
}

int check_subspace(const copes_subspace *S, const char *who) {
  if (!S) return fail(COPES_ERR_INVALID_ARG, "%s: subspace is NULL", who);
  if (S->gathered && S->kind != COPES_SUBSPACE_INDICES)
    return fail(COPES_ERR_INVALID_ARG, "%s: a gathered master needs an INDICES subspace", who);
  if (S->replay_mask && S->kind != COPES_SUBSPACE_HASH_REPLAY)
    return fail(COPES_ERR_INVALID_ARG, "%s: a replay mask needs a HASH_REPLAY subspace", who);
  if (!aligned(S->replay_mask, 16))
    return fail(COPES_ERR_ALIGNMENT, "%s: replay_mask must be 16-byte aligned", who);
  if (!aligned(S->gathered, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: gathered must be 16-byte aligned", who);
  if (S->kind == COPES_SUBSPACE_TILES) {
    if (S->n_tiles && !S->tiles) return fail(COPES_ERR_INVALID_ARG, "%s: tiles is NULL", who);
    if (!aligned(S->tiles, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: tiles must be 16-byte aligned", who);
    if (S->n_tiles > 0x7FFFFFFFull) return fail(COPES_ERR_SIZE, "%s: more than 2^31-1 tiles", who);
    return COPES_OK;
  }
  if (S->kind == COPES_SUBSPACE_INDICES) {
    if (S->n_index && !S->index) return fail(COPES_ERR_INVALID_ARG, "%s: index is NULL", who);
    if (!aligned(S->index, 16))
      return fail(COPES_ERR_ALIGNMENT, "%s: index list must be 16-byte aligned", who);
    if ((S->n_index + copes::kIndexSegment - 1) / copes::kIndexSegment > 0x7FFFFFFFull)
      return fail(COPES_ERR_SIZE, "%s: index list too long", who);
    return COPES_OK;
  }
  if (S->kind == COPES_SUBSPACE_HASH_REPLAY) {
    if (!S->replay) return fail(COPES_ERR_INVALID_ARG, "%s: replay table is NULL", who);
    if (!aligned(S->replay, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: replay table must be 16-byte aligned", who);
    if (S->n_replay_tensors < 1 || S->n_replay_tiles < 1)
      return fail(COPES_ERR_INVALID_ARG, "%s: empty replay table", who);
    if (S->n_replay_tiles > 0x7FFFFFFFull) return fail(COPES_ERR_SIZE, "%s: more than 2^31-1 hash tiles", who);
    if (S->K < 1 || S->K > COPES_MAX_K || S->k < 0 || S->k >= S->K)
      return fail(COPES_ERR_INVALID_ARG, "%s: replay subspace needs 1 <= K <= %d and 0 <= k < K", who,
                  COPES_MAX_K);
    return COPES_OK;
  }
  return fail(COPES_ERR_INVALID_ARG, "%s: unknown subspace kind %d", who, S->kind);
}

size_t replay_map_offset(int n_tensors) { return ((size_t)n_tensors * sizeof(copes::HashTensor) + 15) / 16 * 16; }

copes::ReplayArgs replay_args(const copes_subspace *S) {
  copes::ReplayArgs r{};
  r.table = static_cast<const copes::HashTensor *>(S->replay);
  r.tile_tensor = reinterpret_cast<const uint32_t *>(static_cast<const char *>(S->replay) +
                                                     replay_map_offset(S->n_replay_tensors));
  r.n_tensors = S->n_replay_tensors;
  r.n_tiles = S->n_replay_tiles;
  r.seed_lo = (uint32_t)S->seed;
  r.seed_hi = (uint32_t)(S->seed >> 32);
  r.K = S->K;
  r.k = S->k;
  // floor(x K / 2^32) == k  <=>  ceil(k 2^32 / K) <= x < ceil((k + 1) 2^32 / K)
  const uint64_t lo = (((uint64_t)S->k << 32) + (uint64_t)S->K - 1) / (uint64_t)S->K;
  const uint64_t hi = (((uint64_t)(S->k + 1) << 32) + (uint64_t)S->K - 1) / (uint64_t)S->K;
  r.lo = (uint32_t)lo;
  r.span = (uint32_t)(hi - lo - 1);
  copes::philox_round_keys(r.seed_lo, r.seed_hi, r.rk);
  r.mask = S->replay_mask;
  return r;
}

int check_layout(const copes_layout_desc *L, const char *who) {
  if (!L) return fail(COPES_ERR_INVALID_ARG, "%s: layout is NULL", who);
  if (L->n_tensors <= 0 || !L->numel)
    return fail(COPES_ERR_INVALID_ARG, "%s: layout needs n_tensors > 0 and numel", who);
  return COPES_OK;
}

std::vector<uint64_t> offsets_of(const copes_layout_desc *L) {
  std::vector<uint64_t> off(L->n_tensors + 1, 0);
  for (int t = 0; t < L->n_tensors; ++t) off[t + 1] = (off[t] + L->numel[t] + 63) / 64 * 64;
  return off;
}

using Ranges = std::vector<std::pair<uint64_t, uint64_t>>;

void add_range(Ranges &r, uint64_t b, uint64_t e) {
  if (b >= e) return;
  if (!r.empty() && r.back().second == b) r.back().second = e;
  else r.emplace_back(b, e);
}

int launch_status(cudaError_t e, const char *who) {
  return e == cudaSuccess ? COPES_OK : cuda_fail(e, who);
}

ElemArgs elem_args(const copes_params *p, const copes_subspace *S) {
  ElemArgs a{};
  a.w = p->w;
  a.copies = working_copies(p);
  a.master = p->master;
  a.n_alloc = p->n_alloc;
  if (S->kind == COPES_SUBSPACE_TILES) {
    a.tiles = S->tiles;
    a.n_tiles = S->n_tiles;
  } else {
    a.index = S->index;
    a.n_index = S->n_index;
    a.gathered = S->kind == COPES_SUBSPACE_INDICES ? S->gathered : nullptr;
  }
  return a;
}

// R's coefficients times scale, plus the packed (c, c) pairs of the central polynomial.
void scaled_coeffs(float scale, copes::ScaledCoeffs &k) {
  static const float central[] = COPES_NORMAL_CENTRAL_COEFFS;
  static const float tail[] = COPES_NORMAL_TAIL_COEFFS;
  for (int i = 0; i <= COPES_NORMAL_CENTRAL_DEGREE; ++i) {
    k.central[i] = scale * central[i];
    uint32_t bits;
    memcpy(&bits, &k.central[i], 4);
    k.central2[i] = (unsigned long long)bits | ((unsigned long long)bits << 32);
  }
  for (int i = 0; i <= COPES_NORMAL_TAIL_DEGREE; ++i) k.tail[i] = scale * tail[i];
}

// The antithetic partner buffer (copes_perturb_pair / copes_perturb_partner).
struct Partner {
  const void *buf = nullptr;
  uint64_t base = 0, len = 0;
};

int run_elementwise(int op, const copes_params *p, const copes_subspace *S, uint64_t seed,
                    uint32_t tag, float a_val, float b_val, cudaStream_t s, const char *who,
                    const Partner &partner = Partner{}, uint64_t seed_b = 0) {
  int rc = check_params(p, who);
  if (rc) return rc;
  if ((rc = check_subspace(S, who))) return rc;
  ElemArgs a = elem_args(p, S);
  a.partner = const_cast<void *>(partner.buf);
  a.partner_base = partner.base;
  a.partner_len = partner.len;
  a.seed_lo = (uint32_t)seed;
  a.seed_hi = (uint32_t)(seed >> 32);
  a.tag = tag;
  a.a = a_val;
  a.b = b_val;
  // the scale folded into the normal's polynomial: a * eps = x * (a * R(L))
  scaled_coeffs(a_val, a.coeffs);
  copes::philox_round_keys(a.seed_lo, a.seed_hi, a.rk);
  if (op == copes::kOpPerturbTwoPairs) {
    copes::philox_round_keys((uint32_t)seed_b, (uint32_t)(seed_b >> 32), a.rk_b);
    copes::philox_folded_keys(a.rk, tag, a.fk);
    copes::philox_folded_keys(a.rk_b, tag, a.fk_b);
  }
  if (S->kind == COPES_SUBSPACE_HASH_REPLAY)
    return launch_status(copes::launch_replay_elementwise(op, p->dtype, a, replay_args(S), s), who);
  return launch_status(copes::launch_elementwise(op, S->kind, p->dtype, a, s), who);
}

int split_tiles(const Ranges &r, uint64_t tile_size, std::vector<uint64_t> &tiles) {
  tiles.clear();
  for (const auto &x : r)
    for (uint64_t b = x.first; b < x.second; b += tile_size) {
      tiles.push_back(b);
      tiles.push_back(std::min(b + tile_size, x.second));
    }
  return COPES_OK;
}

// Writes the tile table of r on `stream`.  Up to kTileRangesMax ranges, a kernel expands
// them on the device from its launch parameters: no host copy of the table, which from
// pageable memory can make the host wait for the stream.  Longer range lists (random
// chunks) are split on the host and copied.
int emit_tiles(const Ranges &r, uint64_t tile_size, uint64_t *tiles, uint64_t capacity,
               uint64_t *count, cudaStream_t s, const char *who) {
  uint64_t n = 0;
  for (const auto &x : r) n += (x.second - x.first + tile_size - 1) / tile_size;
  *count = n;
  if (!tiles) return COPES_OK;
  if (capacity < n) return fail(COPES_ERR_WORKSPACE, "%s: %llu tiles needed, capacity %llu", who,
                                (unsigned long long)n, (unsigned long long)capacity);
  if (!aligned(tiles, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: tiles must be 16-byte aligned", who);
  if (n == 0) return COPES_OK;
  if (r.size() <= (size_t)copes::kTileRangesMax) {
    static thread_local copes::TileRanges tr;  // 24 KB: kept off the stack
    tr.n_ranges = (int)r.size();
    tr.tile_size = tile_size;
    uint64_t first = 0;
    for (size_t i = 0; i < r.size(); ++i) {
      tr.begin[i] = r[i].first;
      tr.end[i] = r[i].second;
      tr.first[i] = first;
      first += (r[i].second - r[i].first + tile_size - 1) / tile_size;
    }
    tr.first[r.size()] = first;
    return launch_status(copes::launch_tile_expand(tr, tiles, s), who);
  }
  std::vector<uint64_t> host;
  split_tiles(r, tile_size, host);
  // Pageable source: the call returns once the data is staged, so `host` may go away.
  return launch_status(cudaMemcpyAsync(tiles, host.data(), n * 16, cudaMemcpyHostToDevice, s), who);
}

}  // namespace

void copes::set_last_error(const char *message) { g_message = message; }

extern "C" {

const char *copes_version(void) { return "copes-gb300 0.2 (sm_103a)"; }

int copes_last_error(char *buf, size_t len) {
  if (buf && len) {
    const size_t n = std::min(len - 1, g_message.size());
    memcpy(buf, g_message.data(), n);
    buf[n] = '\0';
  }
  return (int)g_message.size();
}

int copes_check(cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "copes_check");
  const unsigned bits = copes::read_and_clear_es_errors() | copes::read_and_clear_partition_errors() |
                        copes::read_and_clear_replay_errors() | copes::read_and_clear_backup_errors();
  if ((e = cudaGetLastError()) != cudaSuccess) return cuda_fail(e, "copes_check");
  if (bits)
    return fail(COPES_ERR_DEVICE_CHECK,
                "copes_check: a kernel's own check failed and it skipped the work (bits 0x%x: 1 = tile "
                "outside the arena, 2 = gather index outside the arena, 4 = inconsistent partition "
                "workspace or replay table, 8 = a bulk-copy wait ran out, 16 = an element outside "
                "the partner buffer)",
                bits);
  return COPES_OK;
}

int copes_layout(const copes_layout_desc *layout, uint64_t *offsets) {
  int rc = check_layout(layout, "copes_layout");
  if (rc) return rc;
  if (!offsets) return fail(COPES_ERR_INVALID_ARG, "copes_layout: offsets is NULL");
  const std::vector<uint64_t> off = offsets_of(layout);
  std::copy(off.begin(), off.end(), offsets);
  return COPES_OK;
}

double copes_sigma_eff(double sigma, double d, double d_k, int dimension_aware) {
  return dimension_aware ? sigma * sqrt(d / d_k) : sigma;
}

double copes_step_coef(double alpha, int n_members, double sigma_eff, int convention) {
  return convention == COPES_COEF_PAPER ? alpha / (double)n_members
                                        : alpha / ((double)n_members * sigma_eff);
}

int copes_member_table(int n_members, int pairing, int32_t *noise_id, int8_t *sign) {
  if (n_members <= 0 || n_members > COPES_MAX_MEMBERS || !noise_id || !sign)
    return fail(COPES_ERR_INVALID_ARG, "copes_member_table: need 1 <= n_members <= %d and outputs",
                COPES_MAX_MEMBERS);
  if (pairing == COPES_ANTITHETIC) {
    if (n_members % 2) return fail(COPES_ERR_INVALID_ARG, "copes_member_table: antithetic needs even N");
    for (int i = 0; i < n_members; ++i) {
      noise_id[i] = i / 2;
      sign[i] = (i & 1) ? -1 : 1;
    }
    return n_members / 2;
  }
  if (pairing != COPES_ONE_SIDED) return fail(COPES_ERR_INVALID_ARG, "copes_member_table: pairing");
  for (int i = 0; i < n_members; ++i) {
    noise_id[i] = i;
    sign[i] = 1;
  }
  return n_members;
}

uint64_t copes_member_seed(uint64_t base_seed, uint32_t iter, uint32_t k, uint32_t j) {
  uint32_t x[4];
  copes::philox4x32_10(j, k, iter, COPES_TAG_SEED, (uint32_t)base_seed, (uint32_t)(base_seed >> 32), x);
  return (uint64_t)x[0] | ((uint64_t)x[1] << 32);
}

int copes_tiles_from_ranges(const uint64_t *begin, const uint64_t *end, int n_ranges,
                            uint64_t tile_size, uint64_t *tiles, uint64_t capacity,
                            uint64_t *count, cudaStream_t stream) {
  const char *who = "copes_tiles_from_ranges";
  if (n_ranges < 0 || (n_ranges && (!begin || !end)) || !count)
    return fail(COPES_ERR_INVALID_ARG, "%s: bad range arrays", who);
  if (tile_size == 0 || tile_size > (uint64_t)COPES_TILE_MAX)
    return fail(COPES_ERR_SIZE, "%s: tile_size must be in [1, %d]", who, COPES_TILE_MAX);
  Ranges r;
  for (int i = 0; i < n_ranges; ++i) {
    if (begin[i] > end[i]) return fail(COPES_ERR_INVALID_ARG, "%s: range %d has begin > end", who, i);
    add_range(r, begin[i], end[i]);
  }
  return emit_tiles(r, tile_size, tiles, capacity, count, stream, who);
}

int copes_subspace_build(const copes_layout_desc *layout, const copes_partition_spec *spec,
                         int k, uint64_t tile_size, const uint32_t *chunk_map, uint64_t *tiles,
                         uint64_t capacity, uint64_t *count, cudaStream_t stream) {
  const char *who = "copes_subspace_build";
  int rc = check_layout(layout, who);
  if (rc) return rc;
  if (!spec || !count) return fail(COPES_ERR_INVALID_ARG, "%s: spec and count are required", who);
  if (spec->K < 1 || k < 0 || k >= spec->K)
    return fail(COPES_ERR_INVALID_ARG, "%s: need K >= 1 and 0 <= k < K (K=%d, k=%d)", who, spec->K, k);
  if (tile_size == 0 || tile_size > (uint64_t)COPES_TILE_MAX)
    return fail(COPES_ERR_SIZE, "%s: tile_size must be in [1, %d]", who, COPES_TILE_MAX);
  const std::vector<uint64_t> off = offsets_of(layout);
  const int n = layout->n_tensors;
  Ranges r;
  if (spec->mode == COPES_PART_CONTIGUOUS) {
    uint64_t total = 0;
    for (int t = 0; t < n; ++t) total += layout->numel[t];
    const unsigned __int128 T = total;
    const uint64_t lo = (uint64_t)(T * (unsigned)k / (unsigned)spec->K);
    const uint64_t hi = (uint64_t)(T * (unsigned)(k + 1) / (unsigned)spec->K);
    uint64_t rank = 0;
    for (int t = 0; t < n; ++t) {
      const uint64_t a = rank, b = rank + layout->numel[t];
      const uint64_t s = std::max(a, lo), e = std::min(b, hi);
      if (s < e) add_range(r, off[t] + (s - a), off[t] + (e - a));
      rank = b;
    }
  } else if (spec->mode == COPES_PART_TENSOR_GROUPS) {
    if (!spec->group_of) return fail(COPES_ERR_INVALID_ARG, "%s: TENSOR_GROUPS needs group_of", who);
    for (int t = 0; t < n; ++t)
      if (spec->group_of[t] == k) add_range(r, off[t], off[t] + layout->numel[t]);
  } else if (spec->mode == COPES_PART_RANDOM_CHUNKS) {
    const uint64_t C = spec->chunk;
    if (C < 64 || C % 64) return fail(COPES_ERR_INVALID_ARG, "%s: chunk must be a multiple of 64", who);
    if (!chunk_map) return fail(COPES_ERR_INVALID_ARG, "%s: RANDOM_CHUNKS needs the chunk map", who);
    const uint64_t n_chunks = (off[n] + C - 1) / C;
    std::vector<uint32_t> map(n_chunks);
    cudaError_t e = cudaMemcpyAsync(map.data(), chunk_map, n_chunks * 4, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e, who);
    for (int t = 0; t < n; ++t) {
      const uint64_t a = off[t], b = off[t] + layout->numel[t];
      for (uint64_t c = a / C; c * C < b; ++c) {
        if (map[c] != (uint32_t)k) continue;
        add_range(r, std::max(c * C, a), std::min((c + 1) * C, b));
      }
    }
  } else if (spec->mode == COPES_PART_HASH) {
    return fail(COPES_ERR_INVALID_ARG, "%s: HASH partitions are index lists: use copes_hash_count "
                "and copes_hash_fill", who);
  } else {
    return fail(COPES_ERR_INVALID_ARG, "%s: unknown partition mode %d", who, spec->mode);
  }
  return emit_tiles(r, tile_size, tiles, capacity, count, stream, who);
}

size_t copes_random_chunk_map_workspace_bytes(uint64_t n_chunks) {
  if (n_chunks == 0 || n_chunks > (1ull << 20)) return 0;
  return (size_t)copes::chunk_sort_size(n_chunks) * 8;
}

int copes_random_chunk_map(uint64_t n_chunks, int K, uint64_t seed, uint32_t *map, void *workspace,
                           size_t workspace_bytes, cudaStream_t stream) {
  const char *who = "copes_random_chunk_map";
  if (n_chunks == 0 || n_chunks > (1ull << 20))
    return fail(COPES_ERR_SIZE, "%s: n_chunks must be in [1, 2^20]", who);
  if (K < 1) return fail(COPES_ERR_INVALID_ARG, "%s: K must be >= 1", who);
  if (!map) return fail(COPES_ERR_INVALID_ARG, "%s: map is NULL", who);
  const size_t need = copes_random_chunk_map_workspace_bytes(n_chunks);
  if (!workspace || workspace_bytes < need)
    return fail(COPES_ERR_WORKSPACE, "%s: a workspace of %zu bytes is needed", who, need);
  if (!aligned(workspace, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: workspace must be 16-byte aligned", who);
  return launch_status(copes::launch_random_chunk_map(n_chunks, K, seed, map,
                                                      static_cast<uint64_t *>(workspace), stream), who);
}

// ----------------------------------------------------------------------- hash partition
namespace {

struct HashPlan {
  std::vector<copes::HashTensor> tensors;
  uint64_t n_htiles = 0;
  size_t table_bytes = 0, hist_bytes = 0, off_bytes = 0, tot_bytes = 0;
  size_t total() const { return table_bytes + hist_bytes + off_bytes + tot_bytes; }
};

size_t round16(size_t x) { return (x + 15) / 16 * 16; }

HashPlan plan_hash(const copes_layout_desc *L, int K) {
  HashPlan p;
  const std::vector<uint64_t> off = offsets_of(L);
  for (int t = 0; t < L->n_tensors; ++t) {
    if (L->numel[t] == 0) continue;
    copes::HashTensor h{};
    h.offset = off[t];
    h.numel = L->numel[t];
    h.tile_begin = p.n_htiles;
    h.tensor_id = L->tensor_id ? L->tensor_id[t] : (uint32_t)t;
    p.tensors.push_back(h);
    p.n_htiles += (L->numel[t] + copes::kHashTile - 1) / copes::kHashTile;
  }
  p.table_bytes = round16(p.tensors.size() * sizeof(copes::HashTensor));
  p.hist_bytes = round16(p.n_htiles * (size_t)K * 4);
  p.off_bytes = round16(p.n_htiles * (size_t)K * 8);
  p.tot_bytes = round16((size_t)K * 8);
  return p;
}

int check_hash_args(const copes_layout_desc *L, int K, void *ws, size_t ws_bytes, const char *who,
                    HashPlan &plan) {
  int rc = check_layout(L, who);
  if (rc) return rc;
  if (K < 1 || K > COPES_MAX_K) return fail(COPES_ERR_INVALID_ARG, "%s: K must be in [1, %d]", who, COPES_MAX_K);
  plan = plan_hash(L, K);
  if (plan.tensors.empty()) return fail(COPES_ERR_SIZE, "%s: the layout has no elements", who);
  if (plan.n_htiles > 0x7FFFFFFFull) return fail(COPES_ERR_SIZE, "%s: layout too large", who);
  if (!ws || ws_bytes < plan.total())
    return fail(COPES_ERR_WORKSPACE, "%s: workspace of %zu bytes needed", who, plan.total());
  if (!aligned(ws, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: workspace must be 16-byte aligned", who);
  return COPES_OK;
}

}  // namespace

size_t copes_hash_workspace_bytes(const copes_layout_desc *layout, int K) {
  if (!layout || layout->n_tensors <= 0 || !layout->numel || K < 1 || K > COPES_MAX_K) return 0;
  return plan_hash(layout, K).total();
}

int copes_hash_count(const copes_layout_desc *layout, int K, uint64_t seed, void *workspace,
                     size_t workspace_bytes, uint64_t *counts, cudaStream_t stream) {
  const char *who = "copes_hash_count";
  HashPlan plan;
  int rc = check_hash_args(layout, K, workspace, workspace_bytes, who, plan);
  if (rc) return rc;
  if (!counts) return fail(COPES_ERR_INVALID_ARG, "%s: counts is NULL", who);
  char *ws = static_cast<char *>(workspace);
  auto *table = reinterpret_cast<copes::HashTensor *>(ws);
  auto *hist = reinterpret_cast<uint32_t *>(ws + plan.table_bytes);
  auto *totals = reinterpret_cast<unsigned long long *>(ws + plan.table_bytes + plan.hist_bytes + plan.off_bytes);
  cudaError_t e = cudaMemcpyAsync(table, plan.tensors.data(), plan.tensors.size() * sizeof(copes::HashTensor),
                                  cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(totals, 0, (size_t)K * 8, stream);
  if (e == cudaSuccess)
    e = copes::launch_hash_hist(table, (int)plan.tensors.size(), plan.n_htiles, K, seed, hist, totals, stream);
  std::vector<unsigned long long> host(K);
  if (e == cudaSuccess) e = cudaMemcpyAsync(host.data(), totals, (size_t)K * 8, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, who);
  for (int k = 0; k < K; ++k) counts[k] = host[k];
  return COPES_OK;
}

int copes_hash_fill(const copes_layout_desc *layout, int K, uint64_t seed, void *workspace,
                    size_t workspace_bytes, int64_t *const *lists, cudaStream_t stream) {
  const char *who = "copes_hash_fill";
  HashPlan plan;
  int rc = check_hash_args(layout, K, workspace, workspace_bytes, who, plan);
  if (rc) return rc;
  if (!lists) return fail(COPES_ERR_INVALID_ARG, "%s: lists is NULL", who);
  char *ws = static_cast<char *>(workspace);
  auto *table = reinterpret_cast<copes::HashTensor *>(ws);
  auto *hist = reinterpret_cast<uint32_t *>(ws + plan.table_bytes);
  auto *offsets = reinterpret_cast<uint64_t *>(ws + plan.table_bytes + plan.hist_bytes);
  cudaError_t e = copes::launch_hash_scan(hist, plan.n_htiles, K, offsets, stream);
  if (e == cudaSuccess)
    e = copes::launch_hash_scatter(table, (int)plan.tensors.size(), plan.n_htiles, K, seed, offsets,
                                   lists, stream);
  return launch_status(e, who);
}

size_t copes_hash_replay_bytes(const copes_layout_desc *layout) {
  if (!layout || layout->n_tensors <= 0 || !layout->numel) return 0;
  const HashPlan plan = plan_hash(layout, 1);
  return plan.table_bytes + round16(plan.n_htiles * 4);
}

int copes_hash_replay_subspace(const copes_layout_desc *layout, int K, uint64_t seed, int k,
                               void *table, size_t table_bytes, cudaStream_t stream,
                               copes_subspace *out) {
  const char *who = "copes_hash_replay_subspace";
  int rc = check_layout(layout, who);
  if (rc) return rc;
  if (K < 1 || K > COPES_MAX_K) return fail(COPES_ERR_INVALID_ARG, "%s: K must be in [1, %d]", who, COPES_MAX_K);
  if (k < 0 || k >= K) return fail(COPES_ERR_INVALID_ARG, "%s: k must be in [0, K)", who);
  if (!out) return fail(COPES_ERR_INVALID_ARG, "%s: out is NULL", who);
  const HashPlan plan = plan_hash(layout, K);
  if (plan.tensors.empty()) return fail(COPES_ERR_SIZE, "%s: the layout has no elements", who);
  if (plan.n_htiles > 0x7FFFFFFFull) return fail(COPES_ERR_SIZE, "%s: layout too large", who);
  const size_t need = plan.table_bytes + round16(plan.n_htiles * 4);
  if (!table || table_bytes < need)
    return fail(COPES_ERR_WORKSPACE, "%s: a table of %zu bytes is needed", who, need);
  if (!aligned(table, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: table must be 16-byte aligned", who);
  std::vector<uint32_t> tile_tensor(plan.n_htiles);
  for (size_t t = 0; t < plan.tensors.size(); ++t) {
    const uint64_t end = t + 1 < plan.tensors.size() ? plan.tensors[t + 1].tile_begin : plan.n_htiles;
    for (uint64_t i = plan.tensors[t].tile_begin; i < end; ++i) tile_tensor[i] = (uint32_t)t;
  }
  // Pageable sources: each copy returns once its data is staged.
  cudaError_t e = cudaMemcpyAsync(table, plan.tensors.data(), plan.tensors.size() * sizeof(copes::HashTensor),
                                  cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(static_cast<char *>(table) + plan.table_bytes, tile_tensor.data(), plan.n_htiles * 4,
                        cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) return cuda_fail(e, who);
  copes_subspace S{};
  S.kind = COPES_SUBSPACE_HASH_REPLAY;
  S.replay = table;
  S.n_replay_tiles = plan.n_htiles;
  S.n_replay_tensors = (int)plan.tensors.size();
  S.K = K;
  S.k = k;
  S.seed = seed;
  *out = S;
  return COPES_OK;
}

// ------------------------------------------------------------------------------ ES steps
int copes_perturb(const copes_params *p, const copes_subspace *S, uint64_t seed,
                  float signed_sigma, cudaStream_t stream) {
  if (!isfinite(signed_sigma)) return fail(COPES_ERR_INVALID_ARG, "copes_perturb: sigma is not finite");
  return run_elementwise(copes::kOpPerturb, p, S, seed, COPES_TAG_NOISE, signed_sigma, 0.0f, stream,
                         "copes_perturb");
}

// The partner buffer: non-NULL, aligned, inside the arena's index range, and disjoint from
// the working weights w it is read into and from the fp32 master the pair perturb reads
// (esize: bytes per working-dtype element; master NULL in the backup mode).
static int check_partner(uint64_t n_alloc, const void *w, const float *master, uint64_t esize, const void *buf,
                         uint64_t base, uint64_t len, const char *who) {
  if (!buf) return fail(COPES_ERR_INVALID_ARG, "%s: the partner buffer is NULL", who);
  if (!aligned(buf, 16)) return fail(COPES_ERR_ALIGNMENT, "%s: the partner buffer must be 16-byte aligned", who);
  if (base % 4) return fail(COPES_ERR_ALIGNMENT, "%s: partner_base must be a multiple of 4", who);
  if (base > n_alloc || len > n_alloc - base)
    return fail(COPES_ERR_SIZE, "%s: [partner_base, partner_base + partner_len) exceeds the arena", who);
  if (overlaps(buf, len * esize, w, n_alloc * esize))
    return fail(COPES_ERR_INVALID_ARG, "%s: the partner buffer overlaps the working weights w", who);
  if (overlaps(buf, len * esize, master, n_alloc * 4))
    return fail(COPES_ERR_INVALID_ARG, "%s: the partner buffer overlaps the master", who);
  return COPES_OK;
}

int copes_perturb_pair(const copes_params *p, const copes_subspace *S, uint64_t seed,
                       float signed_sigma, void *partner, uint64_t partner_base,
                       uint64_t partner_len, cudaStream_t stream) {
  const char *who = "copes_perturb_pair";
  if (!isfinite(signed_sigma)) return fail(COPES_ERR_INVALID_ARG, "%s: sigma is not finite", who);
  int rc = check_params(p, who);
  if (rc) return rc;
  if ((rc = check_partner(p->n_alloc, p->w, p->master, elem_size(p->dtype), partner, partner_base, partner_len, who)))
    return rc;
  return run_elementwise(copes::kOpPerturbPair, p, S, seed, COPES_TAG_NOISE, signed_sigma, 0.0f, stream,
                         who, Partner{partner, partner_base, partner_len});
}

int copes_perturb_partner(const copes_params *p, const copes_subspace *S, const void *partner,
                          uint64_t partner_base, uint64_t partner_len, cudaStream_t stream) {
  const char *who = "copes_perturb_partner";
  int rc = check_params(p, who);
  if (rc) return rc;
  if ((rc = check_partner(p->n_alloc, p->w, p->master, elem_size(p->dtype), partner, partner_base, partner_len, who)))
    return rc;
  return run_elementwise(copes::kOpPartner, p, S, 0, 0, 0.0f, 0.0f, stream, who,
                         Partner{partner, partner_base, partner_len});
}

int copes_perturb_two_pairs(const copes_params *p, const copes_subspace *S, uint64_t seed_a,
                            uint64_t seed_b, float signed_sigma, cudaStream_t stream) {
  const char *who = "copes_perturb_two_pairs";
  if (!isfinite(signed_sigma)) return fail(COPES_ERR_INVALID_ARG, "%s: sigma is not finite", who);
  int rc = check_params(p, who);
  if (rc) return rc;
  if (!p->w4) return fail(COPES_ERR_INVALID_ARG, "%s: needs four working copies (w2, w3 and w4 set)", who);
  if ((rc = check_subspace(S, who))) return rc;
  if (S->kind != COPES_SUBSPACE_TILES) return fail(COPES_ERR_UNSUPPORTED, "%s: TILES subspaces only", who);
  return run_elementwise(copes::kOpPerturbTwoPairs, p, S, seed_a, COPES_TAG_NOISE, signed_sigma, 0.0f, stream,
                         who, Partner{}, seed_b);
}

int copes_restore(const copes_params *p, const copes_subspace *S, cudaStream_t stream) {
  return run_elementwise(copes::kOpRestore, p, S, 0, 0, 0.0f, 0.0f, stream, "copes_restore");
}

int copes_context_commit(const copes_params *p, const copes_subspace *S, cudaStream_t stream) {
  return run_elementwise(copes::kOpRestore, p, S, 0, 0, 0.0f, 0.0f, stream, "copes_context_commit");
}

int copes_hash_replay_mask(const copes_params *p, const copes_subspace *S, cudaStream_t stream) {
  const char *who = "copes_hash_replay_mask";
  int rc = check_params(p, who);
  if (rc) return rc;
  if ((rc = check_subspace(S, who))) return rc;
  if (S->kind != COPES_SUBSPACE_HASH_REPLAY || !S->replay_mask)
    return fail(COPES_ERR_INVALID_ARG, "%s: needs a HASH_REPLAY subspace with replay_mask set", who);
  copes::ReplayArgs r = replay_args(S);
  r.mask = nullptr;  // the kernel hashes
  return launch_status(copes::launch_replay_mask(r, p->n_alloc, S->replay_mask, stream), who);
}

int copes_gather_master(const copes_params *p, const copes_subspace *S, cudaStream_t stream) {
  if (S && (S->kind != COPES_SUBSPACE_INDICES || !S->gathered))
    return fail(COPES_ERR_INVALID_ARG, "copes_gather_master: needs an INDICES subspace with gathered set");
  return run_elementwise(copes::kOpGather, p, S, 0, 0, 0.0f, 0.0f, stream, "copes_gather_master");
}

int copes_scatter_master(const copes_params *p, const copes_subspace *S, cudaStream_t stream) {
  if (S && (S->kind != COPES_SUBSPACE_INDICES || !S->gathered))
    return fail(COPES_ERR_INVALID_ARG, "copes_scatter_master: needs an INDICES subspace with gathered set");
  return run_elementwise(copes::kOpScatter, p, S, 0, 0, 0.0f, 0.0f, stream, "copes_scatter_master");
}

int copes_init_normal(const copes_params *p, const copes_subspace *S, uint64_t seed, float mean,
                      float scale, cudaStream_t stream) {
  return run_elementwise(copes::kOpInit, p, S, seed, COPES_TAG_INIT, scale, mean, stream,
                         "copes_init_normal");
}

int copes_shape_fitness(const float *rewards, int n, const int32_t *group, int mode,
                        float *fitness, cudaStream_t stream) {
  const char *who = "copes_shape_fitness";
  if (!rewards || !fitness) return fail(COPES_ERR_INVALID_ARG, "%s: rewards / fitness is NULL", who);
  if (n < 1 || n > COPES_MAX_MEMBERS) return fail(COPES_ERR_SIZE, "%s: n must be in [1, %d]", who, COPES_MAX_MEMBERS);
  if (mode < COPES_SHAPE_NONE || mode > COPES_SHAPE_CENTERED_RANK)
    return fail(COPES_ERR_INVALID_ARG, "%s: unknown mode %d", who, mode);
  if (mode == COPES_SHAPE_ZSCORE_GROUPED && !group)
    return fail(COPES_ERR_INVALID_ARG, "%s: ZSCORE_GROUPED needs group ids", who);
  return launch_status(copes::launch_shape(rewards, n, group, mode, fitness, stream), who);
}

namespace {

// The update's member arguments: checks them and fills the noise weights' member table
// (CSR, member order kept within each noise id) and the seeds into `a`.
int fill_update_members(UpdateArgs &a, int n_members, const int32_t *noise_id, const int8_t *sign,
                        const float *fitness, int n_noise, const uint64_t *seeds, float coef,
                        const char *who) {
  if (n_members < 1 || n_members > COPES_MAX_MEMBERS)
    return fail(COPES_ERR_SIZE, "%s: n_members must be in [1, %d]", who, COPES_MAX_MEMBERS);
  if (n_noise < 1 || n_noise > COPES_MAX_NOISE)
    return fail(COPES_ERR_SIZE, "%s: n_noise must be in [1, %d]", who, COPES_MAX_NOISE);
  if (!noise_id || !sign || !fitness || !seeds)
    return fail(COPES_ERR_INVALID_ARG, "%s: noise_id, sign, fitness and seeds are required", who);
  if (!isfinite(coef)) return fail(COPES_ERR_INVALID_ARG, "%s: coef is not finite", who);
  a.fitness = fitness;
  a.coef = coef;
  a.n_members = n_members;
  a.n_noise = n_noise;
  std::vector<int> count(n_noise + 1, 0);
  for (int i = 0; i < n_members; ++i) {
    if (noise_id[i] < 0 || noise_id[i] >= n_noise)
      return fail(COPES_ERR_INVALID_ARG, "%s: noise_id[%d] = %d outside [0, %d)", who, i, noise_id[i], n_noise);
    if (sign[i] != 1 && sign[i] != -1)
      return fail(COPES_ERR_INVALID_ARG, "%s: sign[%d] must be +1 or -1", who, i);
    a.sign[i] = sign[i];
    ++count[noise_id[i] + 1];
  }
  for (int j = 0; j < n_noise; ++j) count[j + 1] += count[j];
  for (int j = 0; j <= n_noise; ++j) a.noise_ptr[j] = (uint16_t)count[j];
  std::vector<int> fillp(count.begin(), count.end() - 1);
  for (int i = 0; i < n_members; ++i) a.noise_member[fillp[noise_id[i]]++] = (uint16_t)i;
  for (int j = 0; j < n_noise; ++j) {
    a.seed_lo[j] = (uint32_t)seeds[j];
    a.seed_hi[j] = (uint32_t)(seeds[j] >> 32);
  }
  return COPES_OK;
}

// Backup mode: checks the arguments and resolves the device address of the pinned backup.
int check_backup(const copes_backup_params *p, const copes_subspace *S, const char *who,
                 uint16_t **backup_dev) {
  if (!p) return fail(COPES_ERR_INVALID_ARG, "%s: params is NULL", who);
  if (!p->w || !p->backup) return fail(COPES_ERR_INVALID_ARG, "%s: w or backup is NULL", who);
  if (!aligned(p->w, 16) || !aligned(p->backup, 16))
    return fail(COPES_ERR_ALIGNMENT, "%s: w and backup must be 16-byte aligned", who);
  if (p->n_alloc == 0) return fail(COPES_ERR_SIZE, "%s: n_alloc is 0", who);
  int rc = check_subspace(S, who);
  if (rc) return rc;
  if (S->kind != COPES_SUBSPACE_TILES)
    return fail(COPES_ERR_UNSUPPORTED, "%s: the backup mode takes TILES subspaces only", who);
  cudaPointerAttributes attr{};
  const cudaError_t e = cudaPointerGetAttributes(&attr, p->backup);
  if (e != cudaSuccess) return cuda_fail(e, who);
  if (attr.type != cudaMemoryTypeHost || !attr.devicePointer)
    return fail(COPES_ERR_INVALID_ARG, "%s: backup must be page-locked host memory", who);
  *backup_dev = static_cast<uint16_t *>(attr.devicePointer);
  return COPES_OK;
}

int run_backup_elementwise(int op, const copes_backup_params *p, const copes_subspace *S, uint64_t seed,
                           float sigma, cudaStream_t s, const char *who,
                           const Partner &partner = Partner{}) {
  uint16_t *dev = nullptr;
  int rc = check_backup(p, S, who, &dev);
  if (rc) return rc;
  if (op == copes::kBackupPerturbPair &&
      (rc = check_partner(p->n_alloc, p->w, nullptr, 2, partner.buf, partner.base, partner.len, who)))
    return rc;
  ElemArgs a{};
  a.partner = const_cast<void *>(partner.buf);
  a.partner_base = partner.base;
  a.partner_len = partner.len;
  a.w = p->w;
  a.n_alloc = p->n_alloc;
  a.tiles = S->tiles;
  a.n_tiles = S->n_tiles;
  a.seed_lo = (uint32_t)seed;
  a.seed_hi = (uint32_t)(seed >> 32);
  a.a = sigma;
  scaled_coeffs(sigma, a.coeffs);
  copes::philox_round_keys(a.seed_lo, a.seed_hi, a.rk);
  return launch_status(copes::launch_backup_elementwise(op, a, dev, s), who);
}

}  // namespace

int copes_update(const copes_params *p, const copes_subspace *S, int n_members,
                 const int32_t *noise_id, const int8_t *sign, const float *fitness, int n_noise,
                 const uint64_t *seeds, float coef, int fuse_commit, cudaStream_t stream) {
  const char *who = "copes_update";
  int rc = check_params(p, who);
  if (rc) return rc;
  if ((rc = check_subspace(S, who))) return rc;
  UpdateArgs a{};
  if ((rc = fill_update_members(a, n_members, noise_id, sign, fitness, n_noise, seeds, coef, who))) return rc;
  a.w = p->w;
  a.copies = working_copies(p);
  a.master = p->master;
  a.n_alloc = p->n_alloc;
  if (S->kind == COPES_SUBSPACE_TILES) {
    a.tiles = S->tiles;
    a.n_tiles = S->n_tiles;
  } else {
    a.index = S->index;
    a.n_index = S->n_index;
    a.gathered = S->kind == COPES_SUBSPACE_INDICES ? S->gathered : nullptr;
  }
  a.fuse_commit = fuse_commit ? 1 : 0;
  if (S->kind == COPES_SUBSPACE_HASH_REPLAY)
    return launch_status(copes::launch_replay_update(p->dtype, a, replay_args(S), stream), who);
  return launch_status(copes::launch_update(S->kind, p->dtype, a, stream, 0), who);
}

// ---------------------------------------------------------------------- backup mode
int copes_backup_save(const copes_backup_params *p, const copes_subspace *S, cudaStream_t stream) {
  return run_backup_elementwise(copes::kBackupSave, p, S, 0, 0.0f, stream, "copes_backup_save");
}

int copes_backup_perturb(const copes_backup_params *p, const copes_subspace *S, uint64_t seed,
                         float signed_sigma, cudaStream_t stream) {
  if (!isfinite(signed_sigma)) return fail(COPES_ERR_INVALID_ARG, "copes_backup_perturb: sigma is not finite");
  return run_backup_elementwise(copes::kBackupPerturb, p, S, seed, signed_sigma, stream, "copes_backup_perturb");
}

int copes_backup_perturb_pair(const copes_backup_params *p, const copes_subspace *S, uint64_t seed,
                              float signed_sigma, void *partner, uint64_t partner_base,
                              uint64_t partner_len, cudaStream_t stream) {
  const char *who = "copes_backup_perturb_pair";
  if (!isfinite(signed_sigma)) return fail(COPES_ERR_INVALID_ARG, "%s: sigma is not finite", who);
  return run_backup_elementwise(copes::kBackupPerturbPair, p, S, seed, signed_sigma, stream, who,
                                Partner{partner, partner_base, partner_len});
}

int copes_backup_perturb_partner(const copes_backup_params *p, const copes_subspace *S,
                                 const void *partner, uint64_t partner_base, uint64_t partner_len,
                                 cudaStream_t stream) {
  const char *who = "copes_backup_perturb_partner";
  uint16_t *dev = nullptr;
  int rc = check_backup(p, S, who, &dev);
  if (rc) return rc;
  if ((rc = check_partner(p->n_alloc, p->w, nullptr, 2, partner, partner_base, partner_len, who))) return rc;
  ElemArgs a{};
  a.w = p->w;
  a.n_alloc = p->n_alloc;
  a.tiles = S->tiles;
  a.n_tiles = S->n_tiles;
  a.partner = const_cast<void *>(partner);
  a.partner_base = partner_base;
  a.partner_len = partner_len;
  return launch_status(copes::launch_elementwise(copes::kOpPartner, COPES_SUBSPACE_TILES, COPES_BF16, a, stream),
                       who);
}

int copes_backup_restore(const copes_backup_params *p, const copes_subspace *S, cudaStream_t stream) {
  return run_backup_elementwise(copes::kBackupRestore, p, S, 0, 0.0f, stream, "copes_backup_restore");
}

int copes_backup_update(const copes_backup_params *p, const copes_subspace *S, int n_members,
                        const int32_t *noise_id, const int8_t *sign, const float *fitness, int n_noise,
                        const uint64_t *seeds, float coef, cudaStream_t stream) {
  const char *who = "copes_backup_update";
  UpdateArgs a{};
  int rc = fill_update_members(a, n_members, noise_id, sign, fitness, n_noise, seeds, coef, who);
  if (rc) return rc;
  uint16_t *dev = nullptr;
  if ((rc = check_backup(p, S, who, &dev))) return rc;
  a.w = p->w;
  a.n_alloc = p->n_alloc;
  a.tiles = S->tiles;
  a.n_tiles = S->n_tiles;
  return launch_status(copes::launch_backup_update(a, dev, stream), who);
}

// ----------------------------------------------------------------------------- debug
int copes_debug_philox(uint64_t seed, uint64_t q0, uint64_t n, uint32_t aux, uint32_t tag,
                       uint32_t *out, cudaStream_t stream) {
  if (!out && n) return fail(COPES_ERR_INVALID_ARG, "copes_debug_philox: out is NULL");
  if (!aligned(out, 16)) return fail(COPES_ERR_ALIGNMENT, "copes_debug_philox: out must be 16-byte aligned");
  if (n > (1ull << 36)) return fail(COPES_ERR_SIZE, "copes_debug_philox: n too large");
  return launch_status(copes::launch_debug_philox(seed, q0, n, aux, tag, out, stream), "copes_debug_philox");
}

int copes_debug_normals(uint64_t seed, uint32_t tag, uint64_t g0, uint64_t n, float *out,
                        cudaStream_t stream) {
  if (!out && n) return fail(COPES_ERR_INVALID_ARG, "copes_debug_normals: out is NULL");
  if (n > (1ull << 36)) return fail(COPES_ERR_SIZE, "copes_debug_normals: n too large");
  return launch_status(copes::launch_debug_normals(seed, tag, g0, n, out, stream), "copes_debug_normals");
}

int copes_debug_transform(const uint32_t *words, uint64_t n, float *out, cudaStream_t stream) {
  if ((!out || !words) && n) return fail(COPES_ERR_INVALID_ARG, "copes_debug_transform: NULL array");
  if (n > (1ull << 36)) return fail(COPES_ERR_SIZE, "copes_debug_transform: n too large");
  return launch_status(copes::launch_debug_transform(words, n, out, stream), "copes_debug_transform");
}

}  // extern "C"
