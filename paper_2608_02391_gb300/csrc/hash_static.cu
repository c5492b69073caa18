// Hash partition without any device allocation, for callers that cannot allocate.
//
// copes_hash_count / copes_hash_fill take their scratch (tensor table, per-tile
// histograms, per-tile offsets, totals) from a workspace the caller allocates.  Some
// callers cannot do that: an ES trainer that shares the GPU with a rollout engine which
// reserved nearly all free HBM for its KV cache at start-up, or code running under a
// framework that owns the device memory pool and forbids further cudaMalloc calls.  This
// entry point runs the same kernels on a fixed scratch array that lives in the library
// image itself (a file-scope __device__ array), so it never calls cudaMalloc, cudaFree
// or any allocating routine, on the device or on the host.
//
// Costs and limits: the array (kStaticScratchBytes) is held by every GPU that loads the
// library until the process exits, and layouts whose scratch would not fit are rejected
// with COPES_ERR_SIZE.  All calls share the one array per device, which keeps the last
// call's contents; calls whose GPU work overlaps (other streams, other host threads)
// race on it and must be serialised by the caller.
#include <stdio.h>

#include <mutex>

#include "copes_internal.h"

namespace {

constexpr size_t kStaticScratchBytes = size_t(8) << 20;  // 8 MiB per device
constexpr int kMaxDevices = 64;
constexpr int kTableChunk = 128;  // tensor-table entries staged per host copy

__device__ __align__(256) unsigned char g_hash_scratch[kStaticScratchBytes];

std::mutex g_scratch_mutex;
void *g_scratch_address[kMaxDevices] = {};

int static_fail(int code, const char *msg) {
  copes::set_last_error(msg);  // reported by copes_last_error like every other failure
  return code;
}

// The device address of g_hash_scratch on the current device.  In host code the name
// g_hash_scratch is only a host-side stand-in, so the address is looked up once per
// device (with that device current) and cached.
cudaError_t scratch_address(void **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_address[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_hash_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_address[dev] = p;
  }
  *out = g_scratch_address[dev];
  return cudaSuccess;
}

size_t round16(size_t x) { return (x + 15) / 16 * 16; }

}  // namespace

extern "C" int copes_hash_partition_static(const copes_layout_desc *layout, int K, uint64_t seed,
                                           int64_t *const *lists, const uint64_t *capacity,
                                           uint64_t *counts, cudaStream_t stream) {
  if (!layout || layout->n_tensors <= 0 || !layout->numel || !counts)
    return static_fail(COPES_ERR_INVALID_ARG, "copes_hash_partition_static: layout and counts are required");
  if (K < 1 || K > COPES_MAX_K)
    return static_fail(COPES_ERR_INVALID_ARG, "copes_hash_partition_static: K must be in [1, 64]");
  if (lists && !capacity)
    return static_fail(COPES_ERR_INVALID_ARG, "copes_hash_partition_static: lists need capacities");

  // Plan the scratch: the tensor table, then per hash tile a K-bucket histogram, then per
  // hash tile K exclusive offsets, then K totals -- the layout copes_hash_count uses.
  uint64_t n_htiles = 0;
  int n_entries = 0;
  for (int t = 0; t < layout->n_tensors; ++t) {
    if (layout->numel[t] == 0) continue;
    ++n_entries;
    n_htiles += (layout->numel[t] + copes::kHashTile - 1) / copes::kHashTile;
  }
  if (n_entries == 0) return static_fail(COPES_ERR_SIZE, "copes_hash_partition_static: empty layout");
  const size_t table_bytes = round16((size_t)n_entries * sizeof(copes::HashTensor));
  const size_t hist_bytes = round16((size_t)n_htiles * K * 4);
  const size_t off_bytes = round16((size_t)n_htiles * K * 8);
  const size_t tot_bytes = round16((size_t)K * 8);
  const size_t need = table_bytes + hist_bytes + off_bytes + tot_bytes;
  if (need > kStaticScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "copes_hash_partition_static: this layout needs %zu bytes of scratch; the static "
             "scratch holds %zu (use copes_hash_count / copes_hash_fill with a workspace)",
             need, kStaticScratchBytes);
    return static_fail(COPES_ERR_SIZE, msg);
  }

  void *base = nullptr;
  cudaError_t e = scratch_address(&base);
  if (e != cudaSuccess) return static_fail(COPES_ERR_CUDA, cudaGetErrorString(e));
  char *ws = static_cast<char *>(base);
  auto *table = reinterpret_cast<copes::HashTensor *>(ws);
  auto *hist = reinterpret_cast<uint32_t *>(ws + table_bytes);
  auto *offsets = reinterpret_cast<uint64_t *>(ws + table_bytes + hist_bytes);
  auto *totals = reinterpret_cast<unsigned long long *>(ws + table_bytes + hist_bytes + off_bytes);

  // Tensor table, staged through a stack buffer (a pageable copy returns once staged).
  copes::HashTensor chunk[kTableChunk];
  uint64_t tile_begin = 0, offset = 0;
  int filled = 0, written = 0;
  for (int t = 0; t < layout->n_tensors && e == cudaSuccess; ++t) {
    const uint64_t numel = layout->numel[t];
    if (numel) {
      copes::HashTensor h{};
      h.offset = offset;
      h.numel = numel;
      h.tile_begin = tile_begin;
      h.tensor_id = layout->tensor_id ? layout->tensor_id[t] : (uint32_t)t;
      chunk[filled++] = h;
      tile_begin += (numel + copes::kHashTile - 1) / copes::kHashTile;
    }
    offset = (offset + numel + 63) / 64 * 64;
    if (filled == kTableChunk || (t == layout->n_tensors - 1 && filled)) {
      e = cudaMemcpyAsync(table + written, chunk, filled * sizeof(copes::HashTensor),
                          cudaMemcpyHostToDevice, stream);
      written += filled;
      filled = 0;
    }
  }
  // The totals accumulate with atomics: they must start at zero on every call.
  if (e == cudaSuccess) e = cudaMemsetAsync(totals, 0, (size_t)K * 8, stream);
  if (e == cudaSuccess) e = copes::launch_hash_hist(table, n_entries, n_htiles, K, seed, hist, totals, stream);
  unsigned long long host_totals[COPES_MAX_K];
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(host_totals, totals, (size_t)K * 8, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return static_fail(COPES_ERR_CUDA, cudaGetErrorString(e));
  for (int k = 0; k < K; ++k) counts[k] = host_totals[k];
  if (!lists) return COPES_OK;

  for (int k = 0; k < K; ++k) {
    if (counts[k] > capacity[k] || (counts[k] && !lists[k]))
      return static_fail(COPES_ERR_WORKSPACE,
                         "copes_hash_partition_static: a list is missing or smaller than its count");
  }
  e = copes::launch_hash_scan(hist, n_htiles, K, offsets, stream);
  if (e == cudaSuccess)
    e = copes::launch_hash_scatter(table, n_entries, n_htiles, K, seed, offsets, lists, stream);
  if (e != cudaSuccess) return static_fail(COPES_ERR_CUDA, cudaGetErrorString(e));
  return COPES_OK;
}
