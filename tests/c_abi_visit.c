/* A plain C99 program that runs one ES visit on the GPU through include/copes.h alone:
 * device memory from the CUDA runtime (cudaMalloc), every step of the visit a copes_*
 * call -- copes_subspace_build, N x copes_perturb, copes_restore, copes_shape_fitness,
 * copes_update without the fused commit, then copes_context_commit (Sec. 3.2, Eq. 8,
 * Eq. 5, Eq. 13).  Before the restore it also runs copes_perturb_two_pairs on four working
 * copies (members 0 .. 3 in one pass, Eq. 8).  Inputs come from a host generator; every input and output is dumped
 * as a raw little-endian file into the directory argv[1], and the run's scalars are
 * printed one per line, for tests/test_c_abi_gpu.py to check against the oracle.
 * Exit status: 0 on success, 2 when a copes_* call fails, 3 when a CUDA call fails. */
#include <cuda_runtime_api.h>

#include <inttypes.h>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "copes.h"

#define CK(call)                                                             \
  do {                                                                       \
    const int rc_ = (call);                                                  \
    if (rc_ != COPES_OK) {                                                   \
      char msg_[512];                                                        \
      copes_last_error(msg_, sizeof msg_);                                   \
      fprintf(stderr, "%s returned %d: %s\n", #call, rc_, msg_);             \
      return 2;                                                              \
    }                                                                        \
  } while (0)

#define CU(call)                                                             \
  do {                                                                       \
    const cudaError_t e_ = (call);                                           \
    if (e_ != cudaSuccess) {                                                 \
      fprintf(stderr, "%s failed: %s\n", #call, cudaGetErrorString(e_));     \
      return 3;                                                              \
    }                                                                        \
  } while (0)

/* Input generation only (not the method's noise): a 64-bit LCG and Box-Muller. */
static uint64_t lcg = 12345;
static double uniform01(void) {
  lcg = lcg * 6364136223846793005ull + 1442695040888963407ull;
  return ((double)(lcg >> 11) + 0.5) * (1.0 / 9007199254740992.0);
}
static double gauss(void) {
  const double u = uniform01(), v = uniform01();
  return sqrt(-2.0 * log(u)) * cos(6.283185307179586 * v);
}

static float bf16_to_float(uint16_t b) {
  const uint32_t x = (uint32_t)b << 16;
  float f;
  memcpy(&f, &x, sizeof f);
  return f;
}

static int dump(const char *dir, const char *name, const void *p, size_t bytes) {
  char path[4096];
  snprintf(path, sizeof path, "%s/%s", dir, name);
  FILE *fh = fopen(path, "wb");
  if (!fh) return 1;
  const size_t n = fwrite(p, 1, bytes, fh);
  fclose(fh);
  return n != bytes;
}

enum { N_MEMBERS = 8, K_PARTS = 3, K_VISIT = 1 };

int main(int argc, char **argv) {
  if (argc < 2) {
    fprintf(stderr, "usage: %s OUTPUT_DIR\n", argv[0]);
    return 1;
  }
  const char *dir = argv[1];
  const uint64_t numel[3] = {300001, 4099, 150000};
  const copes_layout_desc layout = {3, numel, NULL};
  uint64_t off[4];
  CK(copes_layout(&layout, off));
  const uint64_t n = off[3];

  /* theta ~ N(0, 0.02^2) on the parameters, 0 on the layout's padding; objective weights c */
  float *theta = calloc(n, sizeof(float));
  double *c = calloc(n, sizeof(double));
  uint16_t *wh = malloc(n * sizeof(uint16_t));
  float *mh = malloc(n * sizeof(float));
  if (!theta || !c || !wh || !mh) return 1;
  for (int t = 0; t < 3; ++t)
    for (uint64_t e = 0; e < numel[t]; ++e) theta[off[t] + e] = (float)(0.02 * gauss());
  for (uint64_t g = 0; g < n; ++g) c[g] = gauss();

  cudaStream_t s;
  CU(cudaStreamCreate(&s));
  void *w;
  float *master, *d_r, *d_f;
  uint64_t *all_tiles, *tiles;
  CU(cudaMalloc(&w, n * sizeof(uint16_t)));
  CU(cudaMalloc((void **)&master, n * sizeof(float)));
  CU(cudaMalloc((void **)&d_r, N_MEMBERS * sizeof(float)));
  CU(cudaMalloc((void **)&d_f, N_MEMBERS * sizeof(float)));
  CU(cudaMemcpy(master, theta, n * sizeof(float), cudaMemcpyHostToDevice));
  const copes_params p = {w, master, n, COPES_BF16, NULL};

  /* the shared context: w = round(theta) over the whole arena */
  const uint64_t b0 = 0, e0 = n;
  uint64_t n_all = 0, n_tiles = 0;
  CK(copes_tiles_from_ranges(&b0, &e0, 1, COPES_TILE_MAX, NULL, 0, &n_all, s));
  CU(cudaMalloc((void **)&all_tiles, 2 * n_all * sizeof(uint64_t)));
  CK(copes_tiles_from_ranges(&b0, &e0, 1, COPES_TILE_MAX, all_tiles, n_all, &n_all, s));
  copes_subspace all;
  memset(&all, 0, sizeof all);
  all.kind = COPES_SUBSPACE_TILES;
  all.tiles = all_tiles;
  all.n_tiles = n_all;
  CK(copes_context_commit(&p, &all, s));

  /* S = subspace 1 of a contiguous 3-way split, tiles of at most 4,096 elements */
  const copes_partition_spec spec = {COPES_PART_CONTIGUOUS, K_PARTS, 0, 0, NULL};
  CK(copes_subspace_build(&layout, &spec, K_VISIT, 4096, NULL, NULL, 0, &n_tiles, s));
  CU(cudaMalloc((void **)&tiles, 2 * n_tiles * sizeof(uint64_t)));
  CK(copes_subspace_build(&layout, &spec, K_VISIT, 4096, NULL, tiles, n_tiles, &n_tiles, s));
  copes_subspace S;
  memset(&S, 0, sizeof S);
  S.kind = COPES_SUBSPACE_TILES;
  S.tiles = tiles;
  S.n_tiles = n_tiles;
  uint64_t *th = malloc(2 * n_tiles * sizeof(uint64_t));
  if (!th) return 1;
  CU(cudaMemcpyAsync(th, tiles, 2 * n_tiles * sizeof(uint64_t), cudaMemcpyDeviceToHost, s));

  /* the population: antithetic pairs, member seeds of (base 33, iteration 0, subspace 1) */
  int32_t nid[N_MEMBERS];
  int8_t sign[N_MEMBERS];
  const int P = copes_member_table(N_MEMBERS, COPES_ANTITHETIC, nid, sign);
  if (P <= 0) return 2;
  uint64_t seeds[N_MEMBERS];
  for (int j = 0; j < P; ++j) seeds[j] = copes_member_seed(33, 0, K_VISIT, (uint32_t)j);
  const float sigma = 1e-3f;

  /* each member: perturb, then its reward = c . w (a linear objective of the live weights) */
  float rewards[N_MEMBERS];
  for (int i = 0; i < N_MEMBERS; ++i) {
    CK(copes_perturb(&p, &S, seeds[nid[i]], (float)sign[i] * sigma, s));
    CU(cudaMemcpyAsync(wh, w, n * sizeof(uint16_t), cudaMemcpyDeviceToHost, s));
    CU(cudaStreamSynchronize(s));
    if (i < 2) {
      char name[64];
      snprintf(name, sizeof name, "w_member%d.bin", i);
      if (dump(dir, name, wh, n * sizeof(uint16_t))) return 1;
    }
    double r = 0.0;
    for (uint64_t g = 0; g < n; ++g) r += c[g] * (double)bf16_to_float(wh[g]);
    rewards[i] = (float)r;
  }
  /* members 0 .. 3 (noise vectors 0 and 1, signs +, -, +, -) in one pass into four
   * working copies, whose context is committed first */
  void *wc[3];
  for (int c = 0; c < 3; ++c) CU(cudaMalloc(&wc[c], n * sizeof(uint16_t)));
  const copes_params p4 = {w, master, n, COPES_BF16, wc[0], wc[1], wc[2]};
  CK(copes_context_commit(&p4, &all, s));
  CK(copes_perturb_two_pairs(&p4, &S, seeds[nid[0]], seeds[nid[2]], (float)sign[0] * sigma, s));
  for (int c = 0; c < 4; ++c) {
    char name[64];
    snprintf(name, sizeof name, "w_two_pairs%d.bin", c);
    CU(cudaMemcpyAsync(wh, c ? wc[c - 1] : w, n * sizeof(uint16_t), cudaMemcpyDeviceToHost, s));
    CU(cudaStreamSynchronize(s));
    if (dump(dir, name, wh, n * sizeof(uint16_t))) return 1;
  }
  for (int c = 0; c < 3; ++c) CU(cudaFree(wc[c]));

  CK(copes_restore(&p, &S, s));
  CU(cudaMemcpyAsync(wh, w, n * sizeof(uint16_t), cudaMemcpyDeviceToHost, s));
  CU(cudaStreamSynchronize(s));
  if (dump(dir, "w_restored.bin", wh, n * sizeof(uint16_t))) return 1;

  /* shaping (Eq. 5), the update (Eq. 13) without the fused commit, then the commit */
  float f[N_MEMBERS];
  CU(cudaMemcpyAsync(d_r, rewards, sizeof rewards, cudaMemcpyHostToDevice, s));
  CK(copes_shape_fitness(d_r, N_MEMBERS, NULL, COPES_SHAPE_ZSCORE, d_f, s));
  CU(cudaMemcpyAsync(f, d_f, sizeof f, cudaMemcpyDeviceToHost, s));
  const float coef = (float)copes_step_coef(5e-4, N_MEMBERS, sigma, COPES_COEF_OPENAI);
  CK(copes_update(&p, &S, N_MEMBERS, nid, sign, d_f, P, seeds, coef, 0, s));
  CU(cudaMemcpyAsync(wh, w, n * sizeof(uint16_t), cudaMemcpyDeviceToHost, s));
  CU(cudaStreamSynchronize(s));
  if (dump(dir, "w_before_commit.bin", wh, n * sizeof(uint16_t))) return 1;
  CK(copes_context_commit(&p, &S, s));
  CK(copes_check(s));
  CU(cudaMemcpy(wh, w, n * sizeof(uint16_t), cudaMemcpyDeviceToHost));
  CU(cudaMemcpy(mh, master, n * sizeof(float), cudaMemcpyDeviceToHost));

  if (dump(dir, "theta.bin", theta, n * sizeof(float)) || dump(dir, "rewards.bin", rewards, sizeof rewards) ||
      dump(dir, "fitness.bin", f, sizeof f) || dump(dir, "master_after.bin", mh, n * sizeof(float)) ||
      dump(dir, "w_after.bin", wh, n * sizeof(uint16_t)) ||
      dump(dir, "tiles.bin", th, 2 * n_tiles * sizeof(uint64_t)))
    return 1;
  printf("n_alloc %" PRIu64 "\n", n);
  printf("n_tiles %" PRIu64 "\n", n_tiles);
  printf("P %d\n", P);
  printf("seeds");
  for (int j = 0; j < P; ++j) printf(" %" PRIu64, seeds[j]);
  printf("\ncoef %.9e\n", (double)coef);

  CU(cudaFree(w));
  CU(cudaFree(master));
  CU(cudaFree(d_r));
  CU(cudaFree(d_f));
  CU(cudaFree(all_tiles));
  CU(cudaFree(tiles));
  CU(cudaStreamDestroy(s));
  free(theta);
  free(c);
  free(wh);
  free(mh);
  free(th);
  return 0;
}
