/*
 * copes_oracle.c -- plain, slow CPU oracle for the CoPES evolution-strategy core.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg load this library.  The product path (the CUDA library) never calls
 * it, and the two share no code: no headers, tables, constants or helpers.
 *
 * Style: every function walks its elements one by one, in the order the method states,
 * in fp64.  Inputs that the method stores in fp32 (the master copy, rewards, sigma, the
 * step coefficient) are widened exactly; each output is rounded once to its storage
 * type (bf16 or fp32, round-to-nearest-even).
 *
 * What each part follows (paper: "Cooperative Coevolution for Resource-Constrained
 * Agentic LLM Post-Training"):
 *   - Philox4x32-10 counter-based generator: Salmon, Moraes, Dror and Shaw, "Parallel
 *     Random Numbers: As Easy as 1, 2, 3" (SC'11).  It realises the paper's seed replay
 *     (Sec. 3.3 "Seed Replay, Chunked Processing, and Weight Backup"; Supp. A.8): a
 *     perturbation is its seed, and its noise is regenerated from (seed, index).
 *   - Gaussian directions eps ~ N(0, I): Eq. 3 and Eq. 8.  The transform from a Philox
 *     word to a normal is this project's choice (the paper is silent): the exact
 *     standard-normal quantile of an odd 23-bit-lattice uniform.
 *   - Perturbation theta + sigma_k * P_k eps: Eq. 8 (Sec. 3.2); antithetic signs +/-.
 *   - Dimension-aware scale sigma_k = sigma * sqrt(d / d_k): Eq. 11.
 *   - Restore / context commit from the fp32 master: Sec. 3.3 weight backup, Supp. A.8
 *     "CPU Weight Backup"; other parameters keep the shared context (Sec. 3.2).
 *   - Reward standardisation with population std: Eq. 5 (standard ES), Eq. 12 (joint),
 *     Sec. 4.4 "Joint Reward Standardization" (independent per-subspace ablation).
 *   - Reward-weighted update: Eq. 6 (standard ES) and Eq. 13 (composed CoPES update),
 *     Algorithm 1.
 *   - Partitions: Eq. 7 (disjoint, covering, equal sizes), Algorithm 1 (sampled each
 *     step), Supp. A.8 "Partition Replay" (chunk-to-subspace map replayed from a seed).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_TAG_NOISE 0u
#define ORACLE_TAG_INIT 1u
#define ORACLE_TAG_PARTITION 2u
#define ORACLE_TAG_SEED 3u
#define ORACLE_TAG_CHUNK 4u

enum { ORACLE_BF16 = 0, ORACLE_FP32 = 1 };
enum {
  ORACLE_SHAPE_NONE = 0,
  ORACLE_SHAPE_ZSCORE = 1,
  ORACLE_SHAPE_ZSCORE_GROUPED = 2,
  ORACLE_SHAPE_CENTERED_RANK = 3
};
enum { ORACLE_ONE_SIDED = 0, ORACLE_ANTITHETIC = 1 };
enum { ORACLE_COEF_PAPER = 0, ORACLE_COEF_OPENAI = 1 };

/* Non-zero once any routine met an input it cannot handle (e.g. a quantile that did
 * not converge).  Tests assert it stays zero. */
static int oracle_fault = 0;
int oracle_fault_flag(void) { return oracle_fault; }
void oracle_clear_fault(void) { oracle_fault = 0; }

/* ------------------------------------------------------------------------------------
 * Philox4x32-10 (SC'11, Sec. 3 "Philox"): ten rounds on a 4-word counter with a 2-word
 * key.  Each round multiplies words 0 and 2 by the two round multipliers (32x32->64
 * bits), the high halves are XORed with the other two counter words and the round key,
 * the low halves pass through, and the key is bumped by the two Weyl constants.
 * ------------------------------------------------------------------------------------ */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    uint64_t prod0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
    uint64_t prod1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0;
    c1 = n1;
    c2 = n2;
    c3 = n3;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

/* The counter layout used everywhere in this project: (low 32 bits of q, high 32 bits
 * of q, aux, tag); the key is (low, high) 32 bits of the 64-bit seed. */
static void words_at(uint64_t seed, uint64_t q, uint32_t aux, uint32_t tag, uint32_t out[4]) {
  uint32_t ctr[4] = {(uint32_t)q, (uint32_t)(q >> 32), aux, tag};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  oracle_philox4x32_10(ctr, key, out);
}

/* Words for n consecutive counters q0, q0+1, ...; out holds 4 words per counter. */
void oracle_philox_stream(uint64_t seed, uint64_t q0, uint64_t n, uint32_t aux, uint32_t tag,
                          uint32_t *out) {
  for (uint64_t i = 0; i < n; ++i) words_at(seed, q0 + i, aux, tag, out + 4 * i);
}

/* ------------------------------------------------------------------------------------
 * Uniform and normal.
 * u(x) = ((x & 0x7FFFFE) | 1) * 2^-23: bits 1..22 of the word, made odd -- an odd
 * multiple of 2^-23, strictly inside (0, 1), so the quantile below is finite.  u and
 * 1 - u are both exact in fp32 and fp64, and the lattice is symmetric about 1/2.
 * ------------------------------------------------------------------------------------ */
double oracle_uniform(uint32_t x) { return ldexp((double)((x & 0x7FFFFEu) | 1u), -23); }

/* Standard-normal quantile Phi^-1(u), solved by Newton's method on the definition
 * Phi(x) = erfc(-x / sqrt 2) / 2, using libm's erf / erfc.
 *   - u > 1/2 uses the symmetry Phi^-1(u) = -Phi^-1(1 - u) (1 - u is exact here).
 *   - 1/4 <= u < 1/2: solve erf(x / sqrt 2) / 2 = u - 1/2 (exact), from x = 0.  The
 *     function is convex and increasing on x < 0 and x = 0 lies right of the root, so
 *     the iterates decrease monotonically to it.
 *   - u < 1/4: solve ln Phi(x) = ln u.  ln Phi is concave and increasing, and the
 *     Chernoff bound Phi(x) <= exp(-x^2/2)/2 puts x0 = -sqrt(-2 ln 2u) left of the root,
 *     so the iterates increase monotonically to it.
 * Iteration stops once a step is below 2^-50 relative or stops shrinking. */
double oracle_normal_quantile(double u) {
  if (!(u > 0.0 && u < 1.0)) {
    oracle_fault = 1;
    return NAN;
  }
  if (u > 0.5) return -oracle_normal_quantile(1.0 - u);
  if (u == 0.5) return 0.0;
  const double inv_sqrt_2pi = 1.0 / sqrt(2.0 * M_PI);
  const double inv_sqrt_2 = 1.0 / sqrt(2.0);
  double x, dx, prev = INFINITY;
  int it;
  if (u >= 0.25) {
    const double delta = u - 0.5;
    x = 0.0;
    for (it = 0; it < 100; ++it) {
      double density = inv_sqrt_2pi * exp(-0.5 * x * x);
      dx = (0.5 * erf(x * inv_sqrt_2) - delta) / density;
      x -= dx;
      if (!(fabs(dx) > 0x1p-50 * fabs(x)) || (it > 2 && fabs(dx) >= prev)) break;
      prev = fabs(dx);
    }
  } else {
    const double log_u = log(u);
    x = -sqrt(-2.0 * log(2.0 * u));
    for (it = 0; it < 100; ++it) {
      double cdf = 0.5 * erfc(-x * inv_sqrt_2);
      double density = inv_sqrt_2pi * exp(-0.5 * x * x);
      dx = (log(cdf) - log_u) * cdf / density;
      x -= dx;
      if (!(fabs(dx) > 0x1p-50 * fabs(x)) || (it > 2 && fabs(dx) >= prev)) break;
      prev = fabs(dx);
    }
  }
  if (it >= 100) oracle_fault = 1;
  return x;
}

void oracle_normal_quantile_array(const double *u, uint64_t n, double *out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = oracle_normal_quantile(u[i]);
}

/* eps_seed[g]: the normal for global parameter index g.  Counter q = g >> 2 gives four
 * words; index g uses word g & 3.  tag separates independent streams (noise, weight
 * initialisation, ...). */
double oracle_noise_at(uint64_t seed, uint32_t tag, uint64_t g) {
  uint32_t w[4];
  words_at(seed, g >> 2, 0u, tag, w);
  return oracle_normal_quantile(oracle_uniform(w[g & 3u]));
}

void oracle_noise(uint64_t seed, uint32_t tag, const uint64_t *g, uint64_t n, double *out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = oracle_noise_at(seed, tag, g[i]);
}

void oracle_noise_range(uint64_t seed, uint32_t tag, uint64_t g0, uint64_t n, double *out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = oracle_noise_at(seed, tag, g0 + i);
}

/* ------------------------------------------------------------------------------------
 * Rounding to the storage types.
 * ------------------------------------------------------------------------------------ */

/* Round half to even of a non-negative value m (m < 2^53). */
static double round_half_even(double m) {
  double fl = floor(m);
  double frac = m - fl;
  if (frac > 0.5) return fl + 1.0;
  if (frac < 0.5) return fl;
  return (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;
}

/* bf16 has 8 significant bits and fp32's exponent range: its quantum in the binade
 * [2^e, 2^(e+1)) is 2^(e-7), and 2^-133 below the smallest normal 2^-126.  x is rounded
 * to the nearest multiple of the quantum (ties to even); results past the largest
 * finite bf16 become infinity.  The returned bits are the top half of the fp32 image. */
uint16_t oracle_bf16_bits(double x) {
  float as_float;
  uint32_t bits;
  if (x != x) return 0x7FC0u;
  double a = fabs(x);
  double rounded;
  if (a == 0.0 || isinf(a)) {
    rounded = a;
  } else {
    int e = ilogb(a);
    if (e < -126) e = -126;
    double quantum = ldexp(1.0, e - 7);
    rounded = round_half_even(a / quantum) * quantum;
    const double max_bf16 = ldexp(255.0, 120); /* (2 - 2^-7) * 2^127 */
    if (rounded > max_bf16) rounded = INFINITY;
  }
  as_float = (float)(x < 0 ? -rounded : rounded);
  memcpy(&bits, &as_float, 4);
  return (uint16_t)(bits >> 16);
}

double oracle_bf16_value(uint16_t b) {
  uint32_t bits = (uint32_t)b << 16;
  float f;
  memcpy(&f, &bits, 4);
  return (double)f;
}

static void store_value(void *w, int dtype, uint64_t g, double x) {
  if (dtype == ORACLE_BF16) {
    ((uint16_t *)w)[g] = oracle_bf16_bits(x);
  } else {
    ((float *)w)[g] = (float)x; /* C's double -> float conversion rounds to nearest even */
  }
}

/* ------------------------------------------------------------------------------------
 * Subspaces S: a list of global-index ranges [begin, end), or a list of global indices.
 * The oracle visits the elements in the listed order.
 * ------------------------------------------------------------------------------------ */
typedef struct {
  int kind; /* 0: ranges, 1: index list */
  int n_ranges;
  const uint64_t *begin;
  const uint64_t *end;
  const int64_t *idx;
  uint64_t n_idx;
} oracle_subspace;

typedef void (*element_fn)(uint64_t g, void *ctx);

static void for_each_element(const oracle_subspace *S, element_fn fn, void *ctx) {
  if (S->kind == 0) {
    for (int r = 0; r < S->n_ranges; ++r)
      for (uint64_t g = S->begin[r]; g < S->end[r]; ++g) fn(g, ctx);
  } else {
    for (uint64_t i = 0; i < S->n_idx; ++i) fn((uint64_t)S->idx[i], ctx);
  }
}

/* ------------------------------------------------------------------------------------
 * Perturb (Eq. 8): w[g] = round(theta[g] + s * sigma_k * eps_j[g]) for g in S; every
 * other element of w is left alone.  signed_sigma carries the antithetic sign s.
 * ------------------------------------------------------------------------------------ */
double oracle_perturbed_exact(double theta, uint64_t seed, float signed_sigma, uint64_t g) {
  return theta + (double)signed_sigma * oracle_noise_at(seed, ORACLE_TAG_NOISE, g);
}

typedef struct {
  void *w;
  int dtype;
  const float *master;
  uint64_t seed;
  float signed_sigma;
} perturb_ctx;

static void perturb_one(uint64_t g, void *p) {
  perturb_ctx *c = (perturb_ctx *)p;
  store_value(c->w, c->dtype, g,
              oracle_perturbed_exact((double)c->master[g], c->seed, c->signed_sigma, g));
}

void oracle_perturb(void *w, int dtype, const float *master, const oracle_subspace *S,
                    uint64_t seed, float signed_sigma) {
  perturb_ctx c = {w, dtype, master, seed, signed_sigma};
  for_each_element(S, perturb_one, &c);
}

/* Sampled form: n (g, theta[g]) pairs -> the stored bits (bf16 in the low 16 bits, or
 * fp32 bits) and the unrounded fp64 value. */
void oracle_perturb_at(uint64_t n, const uint64_t *g, const float *theta, uint64_t seed,
                       float signed_sigma, int dtype, uint32_t *out_bits, double *out_exact) {
  for (uint64_t i = 0; i < n; ++i) {
    double x = oracle_perturbed_exact((double)theta[i], seed, signed_sigma, g[i]);
    if (out_exact) out_exact[i] = x;
    if (dtype == ORACLE_BF16) {
      out_bits[i] = oracle_bf16_bits(x);
    } else {
      float f = (float)x;
      memcpy(&out_bits[i], &f, 4);
    }
  }
}

/* ------------------------------------------------------------------------------------
 * Restore and context commit: w[g] = round(theta[g]) for g in S.  Restore ends a
 * perturbed evaluation (Supp. A.8, backup restored directly, never by subtracting the
 * replayed noise); commit publishes the updated context after Eq. 13.  Same arithmetic.
 * ------------------------------------------------------------------------------------ */
typedef struct {
  void *w;
  int dtype;
  const float *master;
} restore_ctx;

static void restore_one(uint64_t g, void *p) {
  restore_ctx *c = (restore_ctx *)p;
  store_value(c->w, c->dtype, g, (double)c->master[g]);
}

void oracle_restore(void *w, int dtype, const float *master, const oracle_subspace *S) {
  restore_ctx c = {w, dtype, master};
  for_each_element(S, restore_one, &c);
}

void oracle_commit(void *w, int dtype, const float *master, const oracle_subspace *S) {
  oracle_restore(w, dtype, master, S);
}

/* ------------------------------------------------------------------------------------
 * Fitness shaping.
 *   NONE:            f = r.
 *   ZSCORE:          Eq. 5 / Eq. 12 -- mean and population standard deviation over all
 *                    n rewards, f = (r - mean) / std.
 *   ZSCORE_GROUPED:  the same statistics taken separately within each group id (the
 *                    independent per-subspace standardisation of Sec. 4.4).
 *   CENTERED_RANK:   0-based ranks with ties given their average rank, mapped to
 *                    rank / (n - 1) - 1/2 (centred ranks as in OpenAI-ES).
 * When every reward of a pool is equal the standard deviation is zero and the paper's
 * formula is undefined; f is then 0 for that pool (a zero update).  The test for it is
 * exact equality of all rewards, not a threshold.
 * Returns 0, or -1 for an unknown mode / bad size.
 * ------------------------------------------------------------------------------------ */
static void zscore_pool(const float *r, int n, const int32_t *group, int32_t gid, float *f) {
  double sum = 0.0, sq = 0.0;
  int count = 0, all_equal = 1;
  double first = 0.0;
  for (int i = 0; i < n; ++i) {
    if (group && group[i] != gid) continue;
    if (count == 0) first = (double)r[i];
    if ((double)r[i] != first) all_equal = 0;
    sum += (double)r[i];
    ++count;
  }
  double mean = sum / (double)count;
  for (int i = 0; i < n; ++i) {
    if (group && group[i] != gid) continue;
    double dev = (double)r[i] - mean;
    sq += dev * dev;
  }
  double std = sqrt(sq / (double)count);
  for (int i = 0; i < n; ++i) {
    if (group && group[i] != gid) continue;
    f[i] = all_equal ? 0.0f : (float)(((double)r[i] - mean) / std);
  }
}

int oracle_shape_fitness(const float *r, int n, const int32_t *group, int mode, float *f) {
  if (n <= 0) return -1;
  if (mode == ORACLE_SHAPE_NONE) {
    for (int i = 0; i < n; ++i) f[i] = r[i];
    return 0;
  }
  if (mode == ORACLE_SHAPE_ZSCORE) {
    zscore_pool(r, n, NULL, 0, f);
    return 0;
  }
  if (mode == ORACLE_SHAPE_ZSCORE_GROUPED) {
    if (!group) return -1;
    for (int i = 0; i < n; ++i) {
      int seen = 0;
      for (int j = 0; j < i; ++j)
        if (group[j] == group[i]) seen = 1;
      if (!seen) zscore_pool(r, n, group, group[i], f);
    }
    return 0;
  }
  if (mode == ORACLE_SHAPE_CENTERED_RANK) {
    for (int i = 0; i < n; ++i) {
      if (n == 1) {
        f[i] = 0.0f;
        continue;
      }
      int less = 0, equal = 0;
      for (int j = 0; j < n; ++j) {
        if (r[j] < r[i]) ++less;
        if (r[j] == r[i]) ++equal;
      }
      double rank = (double)less + 0.5 * (double)(equal - 1);
      f[i] = (float)(rank / (double)(n - 1) - 0.5);
    }
    return 0;
  }
  return -1;
}

/* ------------------------------------------------------------------------------------
 * Members and seeds.
 *   ANTITHETIC: member 2j -> (noise j, +1), member 2j+1 -> (noise j, -1).
 *   ONE_SIDED:  member i -> (noise i, +1)  (the paper's standard ES, Eq. 3).
 * seed(base, iter, k, j) = the first two Philox words at counter (j, k, iter, SEED tag)
 * under key = base seed; member noise j of subspace k at iteration iter uses it.
 * ------------------------------------------------------------------------------------ */
int oracle_member_table(int n_members, int pairing, int32_t *noise_id, int8_t *sign) {
  if (pairing == ORACLE_ANTITHETIC) {
    if (n_members % 2) return -1;
    for (int i = 0; i < n_members; ++i) {
      noise_id[i] = i / 2;
      sign[i] = (i % 2 == 0) ? 1 : -1;
    }
    return n_members / 2;
  }
  for (int i = 0; i < n_members; ++i) {
    noise_id[i] = i;
    sign[i] = 1;
  }
  return n_members;
}

uint64_t oracle_member_seed(uint64_t base_seed, uint32_t iter, uint32_t k, uint32_t j) {
  uint32_t ctr[4] = {j, k, iter, ORACLE_TAG_SEED};
  uint32_t key[2] = {(uint32_t)base_seed, (uint32_t)(base_seed >> 32)};
  uint32_t w[4];
  oracle_philox4x32_10(ctr, key, w);
  return (uint64_t)w[0] | ((uint64_t)w[1] << 32);
}

/* Eq. 11: sigma_k = sigma * sqrt(d / d_k) (= sqrt(K) sigma for equal sizes). */
double oracle_sigma_eff(double sigma, double d, double d_k, int dimension_aware) {
  return dimension_aware ? sigma * sqrt(d / d_k) : sigma;
}

/* Step coefficient c in theta+ = theta + c * sum_i f_i s_i eps_i.
 *   PAPER  (Eq. 6, Eq. 13): c = alpha / N_k   (alpha set independently of sigma)
 *   OPENAI (theta += alpha / (N sigma) * sum f eps):  c = alpha / (N_k * sigma_k). */
double oracle_step_coef(double alpha, int n_members, double sigma_eff, int convention) {
  if (convention == ORACLE_COEF_PAPER) return alpha / (double)n_members;
  return alpha / ((double)n_members * sigma_eff);
}

/* ------------------------------------------------------------------------------------
 * Update (Eq. 6, Eq. 13): theta[g] += c * sum_i s_i f_i eps_{noise(i)}[g] for g in S.
 * Members sharing a noise vector are first folded into one weight per noise vector,
 * w_j = sum over members i with noise(i) = j of s_i f_i (member order).
 * ------------------------------------------------------------------------------------ */
void oracle_noise_weights(int n_members, const int32_t *noise_id, const int8_t *sign,
                          const float *f, int n_noise, double *wj) {
  for (int j = 0; j < n_noise; ++j) wj[j] = 0.0;
  for (int i = 0; i < n_members; ++i) wj[noise_id[i]] += (double)sign[i] * (double)f[i];
}

/* theta + c * sum_j wj[j] eps_j[g] in fp64; *scale gets |c| * sum_j |wj[j] eps_j[g]|,
 * the magnitude that bounds the rounding error of any fp32 evaluation of the sum. */
double oracle_updated_exact(double theta, uint64_t g, int n_noise, const uint64_t *seeds,
                            const double *wj, double coef, double *scale) {
  double acc = 0.0, mag = 0.0;
  for (int j = 0; j < n_noise; ++j) {
    double e = oracle_noise_at(seeds[j], ORACLE_TAG_NOISE, g);
    acc += wj[j] * e;
    mag += fabs(wj[j] * e);
  }
  if (scale) *scale = fabs(coef) * mag;
  return theta + coef * acc;
}

void oracle_update_at(uint64_t n, const uint64_t *g, const float *theta, int n_noise,
                      const uint64_t *seeds, const double *wj, float coef, float *out_theta,
                      double *out_exact, double *out_scale) {
  for (uint64_t i = 0; i < n; ++i) {
    double scale = 0.0;
    double x = oracle_updated_exact((double)theta[i], g[i], n_noise, seeds, wj, (double)coef,
                                    &scale);
    out_theta[i] = (float)x;
    if (out_exact) out_exact[i] = x;
    if (out_scale) out_scale[i] = scale;
  }
}

typedef struct {
  float *master;
  void *w;
  int dtype;
  int n_noise;
  const uint64_t *seeds;
  const double *wj;
  double coef;
} update_ctx;

static void update_one(uint64_t g, void *p) {
  update_ctx *c = (update_ctx *)p;
  double x = oracle_updated_exact((double)c->master[g], g, c->n_noise, c->seeds, c->wj,
                                  c->coef, NULL);
  c->master[g] = (float)x;
  if (c->w) store_value(c->w, c->dtype, g, (double)c->master[g]);
}

/* w may be NULL; otherwise the context commit w[g] = round(theta+[g]) follows. */
int oracle_update(float *master, void *w, int dtype, const oracle_subspace *S, int n_members,
                  const int32_t *noise_id, const int8_t *sign, const float *f, int n_noise,
                  const uint64_t *seeds, float coef) {
  double *wj = (double *)malloc(sizeof(double) * (size_t)(n_noise > 0 ? n_noise : 1));
  if (!wj) return -1;
  oracle_noise_weights(n_members, noise_id, sign, f, n_noise, wj);
  update_ctx c = {master, w, dtype, n_noise, seeds, wj, (double)coef};
  for_each_element(S, update_one, &c);
  free(wj);
  return 0;
}

/* ------------------------------------------------------------------------------------
 * Parameter layout and subspace construction.
 * Tensors are laid out in order in one global index space; tensor t starts at
 * offsets[t], and offsets[t+1] = offsets[t] + numel[t] rounded up to a multiple of 64.
 * Padding indices belong to no subspace.
 * ------------------------------------------------------------------------------------ */
void oracle_layout(const uint64_t *numel, int n_tensors, uint64_t *offsets) {
  offsets[0] = 0;
  for (int t = 0; t < n_tensors; ++t) offsets[t + 1] = (offsets[t] + numel[t] + 63u) / 64u * 64u;
}

static int push_range(uint64_t b, uint64_t e, uint64_t *begin, uint64_t *end, int count,
                      int max_ranges) {
  if (b >= e) return count;
  if (count > 0 && end[count - 1] == b) {
    end[count - 1] = e;
    return count;
  }
  if (count >= max_ranges) return -1;
  begin[count] = b;
  end[count] = e;
  return count + 1;
}

/* CONTIGUOUS: the parameters, in layout order, cut into K consecutive parts; part k
 * holds the parameters of rank [floor(n k / K), floor(n (k+1) / K)) where n is the
 * number of (non-padding) parameters.  Returns the number of ranges, or -1. */
int oracle_contiguous_ranges(const uint64_t *offsets, const uint64_t *numel, int n_tensors,
                             int K, int k, uint64_t *begin, uint64_t *end, int max_ranges) {
  uint64_t n = 0;
  for (int t = 0; t < n_tensors; ++t) n += numel[t];
  uint64_t lo = (uint64_t)((unsigned __int128)n * (unsigned)k / (unsigned)K);
  uint64_t hi = (uint64_t)((unsigned __int128)n * (unsigned)(k + 1) / (unsigned)K);
  uint64_t rank = 0;
  int count = 0;
  for (int t = 0; t < n_tensors && count >= 0; ++t) {
    uint64_t a = rank, b = rank + numel[t];
    uint64_t s = a > lo ? a : lo, e = b < hi ? b : hi;
    if (s < e) count = push_range(offsets[t] + (s - a), offsets[t] + (e - a), begin, end, count,
                                  max_ranges);
    rank = b;
  }
  return count;
}

/* TENSOR_GROUPS: the union of the tensors whose group id is k, in layout order. */
int oracle_group_ranges(const uint64_t *offsets, const uint64_t *numel, int n_tensors,
                        const int32_t *group_of, int k, uint64_t *begin, uint64_t *end,
                        int max_ranges) {
  int count = 0;
  for (int t = 0; t < n_tensors && count >= 0; ++t)
    if (group_of[t] == k)
      count = push_range(offsets[t], offsets[t] + numel[t], begin, end, count, max_ranges);
  return count;
}

/* HASH: element e of the tensor with id tid goes to subspace
 *   floor(x * K / 2^32), x = word (e & 3) of Philox(seed; e >> 2, tid, PARTITION tag),
 * i.e. a uniform 32-bit hash of (tensor id, element index) scaled to K buckets. */
uint32_t oracle_hash_subspace(uint64_t seed, uint32_t tensor_id, uint64_t e, uint32_t K) {
  uint32_t w[4];
  words_at(seed, e >> 2, tensor_id, ORACLE_TAG_PARTITION, w);
  return (uint32_t)(((uint64_t)w[e & 3u] * (uint64_t)K) >> 32);
}

/* The sorted global-index list of subspace k; out may be NULL to count only. */
uint64_t oracle_hash_list(const uint64_t *offsets, const uint64_t *numel,
                          const uint32_t *tensor_ids, int n_tensors, uint32_t K, uint64_t seed,
                          uint32_t k, int64_t *out) {
  uint64_t count = 0;
  for (int t = 0; t < n_tensors; ++t)
    for (uint64_t e = 0; e < numel[t]; ++e)
      if (oracle_hash_subspace(seed, tensor_ids[t], e, K) == k) {
        if (out) out[count] = (int64_t)(offsets[t] + e);
        ++count;
      }
  return count;
}

/* RANDOM_CHUNKS (Eq. 7 at chunk granularity; Supp. A.8 partition replay): chunk c (the
 * global indices [c C, (c+1) C)) gets the key x0 of Philox(seed; c, 0, CHUNK tag); the
 * chunks are ranked by (key, c), and the chunk of rank r goes to subspace
 * floor(r K / n_chunks).  Every subspace gets floor or ceil of n_chunks / K chunks. */
typedef struct {
  uint32_t key;
  uint64_t chunk;
} chunk_key;

static int cmp_chunk_key(const void *a, const void *b) {
  const chunk_key *x = (const chunk_key *)a, *y = (const chunk_key *)b;
  if (x->key != y->key) return x->key < y->key ? -1 : 1;
  if (x->chunk != y->chunk) return x->chunk < y->chunk ? -1 : 1;
  return 0;
}

int oracle_random_chunks(uint64_t n_chunks, uint32_t K, uint64_t seed, uint32_t *chunk_subspace) {
  chunk_key *keys = (chunk_key *)malloc(sizeof(chunk_key) * (size_t)(n_chunks ? n_chunks : 1));
  if (!keys) return -1;
  for (uint64_t c = 0; c < n_chunks; ++c) {
    uint32_t w[4];
    words_at(seed, c, 0u, ORACLE_TAG_CHUNK, w);
    keys[c].key = w[0];
    keys[c].chunk = c;
  }
  qsort(keys, (size_t)n_chunks, sizeof(chunk_key), cmp_chunk_key);
  for (uint64_t r = 0; r < n_chunks; ++r)
    chunk_subspace[keys[r].chunk] =
        (uint32_t)((unsigned __int128)r * K / (unsigned __int128)n_chunks);
  free(keys);
  return 0;
}

/* The ranges of subspace k under a chunk map, intersected with the tensors (padding
 * excluded).  Returns the number of ranges, or -1 if max_ranges is too small. */
int oracle_chunk_ranges(const uint64_t *offsets, const uint64_t *numel, int n_tensors,
                        uint64_t chunk, const uint32_t *chunk_subspace, uint32_t k,
                        uint64_t *begin, uint64_t *end, int max_ranges) {
  int count = 0;
  for (int t = 0; t < n_tensors && count >= 0; ++t) {
    uint64_t a = offsets[t], b = offsets[t] + numel[t];
    for (uint64_t c = a / chunk; c * chunk < b && count >= 0; ++c) {
      if (chunk_subspace[c] != k) continue;
      uint64_t s = c * chunk > a ? c * chunk : a;
      uint64_t e = (c + 1) * chunk < b ? (c + 1) * chunk : b;
      count = push_range(s, e, begin, end, count, max_ranges);
    }
  }
  return count;
}
