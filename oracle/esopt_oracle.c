/*
 * Plain, slow CPU oracle for the parameter-space ES step of Agentic ESOpt.
 *
 * TEST INFRASTRUCTURE ONLY. Only the test suite, the package smoke check and
 * the CPU-baseline leg of the benchmark may load or call this file. The product
 * path (the CUDA library and its Python binding) never links, imports or calls
 * it, and this file shares no code, header, constant table or helper with that
 * path.
 *
 * Every function here is the definition written out in double precision, one
 * step at a time, in the order the method states it:
 *
 *   - noise:     eps_seed[g] for global parameter index g, regenerated from the
 *                integer seed (the paper stores only the seed; §3 last
 *                paragraph, App. D.6).  The generator itself is not named by
 *                the paper; this build fixes Philox4x32-10 (Salmon et al.,
 *                "Parallel random numbers: as easy as 1, 2, 3", SC'11) keyed by
 *                (seed, index) and the Box-Muller transform (Box & Muller,
 *                1958).
 *   - perturb:   theta <- R(theta + s * eps)              (§3, App. D.6)
 *   - restore:   theta <- R(theta - s * eps)              (§3, App. D.6)
 *   - update:    theta <- R(theta + sum_i c_i * eps_i)    (§3 implemented
 *                update; App. C.1 canonical estimator)
 *   - rewards:   population z-score                       (§3)
 *   - schedule:  cosine decay of sigma                    (§3.1)
 *   - coefficients for the update (paper scale alpha/G and the canonical
 *     alpha/(G sigma) of App. C.1), and the antithetic fold.
 *
 * R is one rounding of the double-precision value to the storage type
 * (round-to-nearest-even for fp32, bf16 and FP8 E4M3; E4M3 saturates at its
 * largest finite value and is stored with a per-segment scale).
 *
 * Parity is pinned against: an independent Philox implementation (PyTorch's
 * host engine), closed forms, invariants and brute-force Monte Carlo checks in
 * the test suite. No function here is "parity unpinned".
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* Philox4x32-10 (SC'11, Philox-4x32 with R = 10 rounds).                     */
/* ------------------------------------------------------------------------- */

/* Round multipliers and Weyl key increments of Philox-4x32 as published. */
static const uint32_t PHILOX_MUL_A = 0xD2511F53u;
static const uint32_t PHILOX_MUL_B = 0xCD9E8D57u;
static const uint32_t PHILOX_WEYL_A = 0x9E3779B9u;
static const uint32_t PHILOX_WEYL_B = 0xBB67AE85u;

/*
 * One Philox-4x32 block: counter (x0, x1, x2, x3) and key (k0, k1) give four
 * 32-bit outputs. Each round multiplies x0 and x2 by the two constants into
 * 64-bit products; the high halves are mixed with the other two words and the
 * round key, the low halves become the new x1 and x3. The key advances by the
 * Weyl increments between rounds.
 */
void oracle_philox4x32_10(const uint32_t counter[4], const uint32_t key[2],
                          uint32_t out[4]) {
  uint32_t x0 = counter[0], x1 = counter[1], x2 = counter[2], x3 = counter[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += PHILOX_WEYL_A;
      k1 += PHILOX_WEYL_B;
    }
    uint64_t prod_a = (uint64_t)PHILOX_MUL_A * (uint64_t)x0;
    uint64_t prod_b = (uint64_t)PHILOX_MUL_B * (uint64_t)x2;
    uint32_t hi_a = (uint32_t)(prod_a >> 32), lo_a = (uint32_t)prod_a;
    uint32_t hi_b = (uint32_t)(prod_b >> 32), lo_b = (uint32_t)prod_b;
    uint32_t y0 = hi_b ^ x1 ^ k0;
    uint32_t y1 = lo_b;
    uint32_t y2 = hi_a ^ x3 ^ k1;
    uint32_t y3 = lo_a;
    x0 = y0;
    x1 = y1;
    x2 = y2;
    x3 = y3;
  }
  out[0] = x0;
  out[1] = x1;
  out[2] = x2;
  out[3] = x3;
}

/*
 * The block that holds parameter index g: block number j = floor(g / 4),
 * counter = (low 32 bits of j, high 32 bits of j, 0, 0),
 * key     = (low 32 bits of seed, high 32 bits of seed).
 */
void oracle_noise_block(uint64_t seed, uint64_t j, uint32_t out[4]) {
  uint32_t counter[4] = {(uint32_t)j, (uint32_t)(j >> 32), 0u, 0u};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  oracle_philox4x32_10(counter, key, out);
}

/*
 * Uniform variate in the open interval (0, 1) from the top 23 bits of a
 * 32-bit output: u = (2 m + 1) / 2^24 with m = x >> 9. The set of values is
 * symmetric about 1/2 and excludes 0 and 1, so log(u) is always finite.
 */
/* Words of blocks j0 .. j0 + n - 1, block after block (4 words each): the
 * same definition as oracle_noise_block, over a range. */
void oracle_noise_blocks(uint64_t seed, uint64_t j0, uint64_t n, uint32_t* out) {
  for (uint64_t k = 0; k < n; ++k) oracle_noise_block(seed, j0 + k, out + 4 * k);
}

double oracle_uniform(uint32_t x) {
  double m = (double)(x >> 9);
  return (2.0 * m + 1.0) / 16777216.0;
}

/*
 * Box-Muller: the pair (u_a, u_b) gives the two standard normals
 * r cos(phi) and r sin(phi), with r = sqrt(-2 ln u_a) and phi = 2 pi u_b.
 * Output words (x0, x1) of a block form the first pair (elements 4j, 4j+1),
 * (x2, x3) the second (elements 4j+2, 4j+3).
 */
void oracle_box_muller(uint32_t x_a, uint32_t x_b, double out[2]) {
  double u_a = oracle_uniform(x_a);
  double u_b = oracle_uniform(x_b);
  double r = sqrt(-2.0 * log(u_a));
  double phi = 2.0 * M_PI * u_b;
  out[0] = r * cos(phi);
  out[1] = r * sin(phi);
}

/* Box-Muller on word pairs: out[2k], out[2k+1] from (words[2k], words[2k+1]). */
void oracle_box_muller_fill(const uint32_t* words, uint64_t npairs, double* out) {
  for (uint64_t k = 0; k < npairs; ++k)
    oracle_box_muller(words[2 * k], words[2 * k + 1], out + 2 * k);
}

double oracle_gaussian(uint64_t seed, uint64_t g) {
  uint32_t x[4];
  oracle_noise_block(seed, g >> 2, x);
  int k = (int)(g & 3u);
  int pair = k >> 1;
  double e[2];
  oracle_box_muller(x[2 * pair], x[2 * pair + 1], e);
  return e[k & 1];
}

/* eps_seed[g] for g in [index_base, index_base + n). */
void oracle_noise_fill(uint64_t seed, uint64_t index_base, uint64_t n,
                       double* out) {
  for (uint64_t k = 0; k < n; ++k) out[k] = oracle_gaussian(seed, index_base + k);
}

/* eps_seed[g[k]] for an arbitrary list of global indices. */
void oracle_noise_at(uint64_t seed, const uint64_t* g, uint64_t n, double* out) {
  for (uint64_t k = 0; k < n; ++k) out[k] = oracle_gaussian(seed, g[k]);
}

/* ------------------------------------------------------------------------- */
/* Storage rounding.                                                          */
/* ------------------------------------------------------------------------- */

/* bf16 bits -> value (bf16 is the top half of an IEEE binary32). */
double oracle_bf16_to_double(uint16_t h) {
  uint32_t bits = (uint32_t)h << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

/*
 * Round a double to the nearest bfloat16 (8 significant bits, binary32
 * exponent range), ties to even, in one step. rint() does the rounding under
 * the default round-to-nearest-even mode. Values at or beyond 2^128 after
 * rounding overflow to infinity; NaN maps to a quiet NaN of the same sign.
 */
uint16_t oracle_bf16_from_double(double x) {
  uint16_t sign = signbit(x) ? 0x8000u : 0x0000u;
  if (isnan(x)) return (uint16_t)(sign | 0x7FC0u);
  if (isinf(x)) return (uint16_t)(sign | 0x7F80u);
  double a = fabs(x);
  double q;
  if (a < 0x1p-126) {
    /* subnormal range: fixed spacing 2^-133 */
    q = rint(a * 0x1p133) * 0x1p-133;
  } else {
    int e;
    frexp(a, &e); /* a = f * 2^e, f in [0.5, 1): top bit has weight 2^(e-1) */
    q = ldexp(rint(ldexp(a, 8 - e)), e - 8);
  }
  if (q >= 0x1p128) return (uint16_t)(sign | 0x7F80u);
  float f = (float)q; /* exact: at most 8 significant bits, in range */
  uint32_t bits;
  memcpy(&bits, &f, sizeof bits);
  return (uint16_t)(sign | (uint16_t)((bits >> 16) & 0x7FFFu));
}

/* Round a double to binary32, ties to even (the C conversion). */
float oracle_f32_from_double(double x) { return (float)x; }

/*
 * FP8 E4M3 storage (the quantized-weight direction the paper leaves as future
 * work, App. A.2; only the storage grid is new, the step is unchanged). The
 * E4M3 format of the OCP 8-bit floating-point specification: 1 sign bit, 4
 * exponent bits with bias 7, 3 mantissa bits; exponent 0 holds the subnormals
 * m * 2^-9; there are no infinities, exponent 15 with mantissa 7 is NaN, and
 * the largest finite magnitude is 1.75 * 2^8 = 448.
 *
 * A segment stored in E4M3 carries one scale s > 0: element k has the value
 * s * e4m3(code[k]).
 */
double oracle_e4m3_to_double(uint8_t c) {
  int exponent = (c >> 3) & 0xF;
  int mantissa = c & 0x7;
  double v;
  if (exponent == 0xF && mantissa == 0x7)
    v = NAN;
  else if (exponent == 0)
    v = mantissa * 0x1p-9;
  else
    v = ldexp(1.0 + mantissa / 8.0, exponent - 7);
  return (c & 0x80) ? -v : v;
}

/*
 * Round a double to the nearest E4M3 value, ties to even, saturating: a
 * magnitude beyond the largest finite value (448), infinities included,
 * becomes 448 with its sign. NaN maps to the NaN code of the same sign.
 */
uint8_t oracle_e4m3_from_double(double x) {
  uint8_t sign = signbit(x) ? 0x80u : 0x00u;
  if (isnan(x)) return (uint8_t)(sign | 0x7Fu);
  double a = fabs(x);
  if (a >= 448.0) return (uint8_t)(sign | 0x7Eu);
  double q;
  if (a < 0x1p-6) {
    /* subnormal range: fixed spacing 2^-9 */
    q = rint(a * 0x1p9) * 0x1p-9;
  } else {
    int e;
    frexp(a, &e); /* a = f * 2^e, f in [0.5, 1): 4 significant bits -> spacing 2^(e-4) */
    q = ldexp(rint(ldexp(a, 4 - e)), e - 4);
  }
  if (q > 448.0) q = 448.0;
  if (q == 0.0) return sign;
  if (q < 0x1p-6) return (uint8_t)(sign | (uint8_t)(q * 0x1p9));
  int e;
  double f = frexp(q, &e); /* q = (2f) 2^(e-1), 2f in [1, 2) */
  int exponent = e - 1 + 7;
  int mantissa = (int)((2.0 * f - 1.0) * 8.0);
  return (uint8_t)(sign | (uint8_t)(exponent << 3) | (uint8_t)mantissa);
}

/* ------------------------------------------------------------------------- */
/* Perturb / restore / update on host arrays.                                 */
/*                                                                           */
/* Each element is identified by its global parameter index g[k]; theta[k]   */
/* is updated in place. "scale" is the signed perturbation s = +sigma       */
/* (perturb) or -sigma (restore) exactly as the float handed to the device. */
/* ------------------------------------------------------------------------- */

void oracle_axpy_noise_f32(float* theta, const uint64_t* g, uint64_t n,
                           uint64_t seed, float scale) {
  for (uint64_t k = 0; k < n; ++k) {
    double v = (double)theta[k] + (double)scale * oracle_gaussian(seed, g[k]);
    theta[k] = oracle_f32_from_double(v);
  }
}

void oracle_axpy_noise_bf16(uint16_t* theta, const uint64_t* g, uint64_t n,
                            uint64_t seed, float scale) {
  for (uint64_t k = 0; k < n; ++k) {
    double v = oracle_bf16_to_double(theta[k]) +
               (double)scale * oracle_gaussian(seed, g[k]);
    theta[k] = oracle_bf16_from_double(v);
  }
}

/* Perturb / restore of an E4M3 segment with scale s: the value s * e4m3(code)
   moves by scale * eps, and the result is stored as the nearest E4M3 code of
   (value / s). */
void oracle_axpy_noise_e4m3(uint8_t* codes, const uint64_t* g, uint64_t n, uint64_t seed,
                            float scale, float seg_scale) {
  const double s = (double)seg_scale;
  for (uint64_t k = 0; k < n; ++k) {
    double v = s * oracle_e4m3_to_double(codes[k]) + (double)scale * oracle_gaussian(seed, g[k]);
    codes[k] = oracle_e4m3_from_double(v / s);
  }
}

/*
 * theta[k] <- R(theta[k] + sum_{i=0}^{nseeds-1} coeffs[i] * eps_{seeds[i]}[g[k]]),
 * the sum taken in double in ascending i, then one rounding.
 */
void oracle_update_f32(float* theta, const uint64_t* g, uint64_t n,
                       const uint64_t* seeds, const float* coeffs, int nseeds) {
  for (uint64_t k = 0; k < n; ++k) {
    double sum = 0.0;
    for (int i = 0; i < nseeds; ++i)
      sum += (double)coeffs[i] * oracle_gaussian(seeds[i], g[k]);
    theta[k] = oracle_f32_from_double((double)theta[k] + sum);
  }
}

void oracle_update_bf16(uint16_t* theta, const uint64_t* g, uint64_t n,
                        const uint64_t* seeds, const float* coeffs, int nseeds) {
  for (uint64_t k = 0; k < n; ++k) {
    double sum = 0.0;
    for (int i = 0; i < nseeds; ++i)
      sum += (double)coeffs[i] * oracle_gaussian(seeds[i], g[k]);
    theta[k] = oracle_bf16_from_double(oracle_bf16_to_double(theta[k]) + sum);
  }
}

/* The update of an E4M3 segment with scale s: value s * e4m3(code) plus the
   reward-weighted sum (double, ascending i), stored as the nearest E4M3 code of
   (value / s). */
void oracle_update_e4m3(uint8_t* codes, const uint64_t* g, uint64_t n, const uint64_t* seeds,
                        const float* coeffs, int nseeds, float seg_scale) {
  const double s = (double)seg_scale;
  for (uint64_t k = 0; k < n; ++k) {
    double sum = 0.0;
    for (int i = 0; i < nseeds; ++i)
      sum += (double)coeffs[i] * oracle_gaussian(seeds[i], g[k]);
    codes[k] = oracle_e4m3_from_double((s * oracle_e4m3_to_double(codes[k]) + sum) / s);
  }
}

/* ------------------------------------------------------------------------- */
/* Host-side generation control.                                              */
/* ------------------------------------------------------------------------- */

/*
 * Population z-score (§3): Rhat_i = (R_i - mu) / (s + eps_z) with
 * mu = (1/G) sum R_j and s^2 = (1/G) sum (R_j - mu)^2.
 *
 * Invalid rewards (§5 and App. D.5/D.6, automatic heuristic design): a
 * non-finite reward is replaced, before normalisation, by a finite penalty
 * drawn from the same batch; this oracle uses its smallest finite reward.
 * A batch with no finite reward, or whose rewards are all equal, produces no
 * update: every Rhat_i is 0.
 *
 * Returns the number of non-finite entries that were replaced, or -1 for an
 * invalid argument.
 */
int oracle_zscore(const double* R, int n, double eps_z, double* Rhat) {
  if (n < 1) return -1;
  int n_finite = 0;
  double lo = 0.0, hi = 0.0;
  for (int i = 0; i < n; ++i) {
    if (!isfinite(R[i])) continue;
    if (n_finite == 0 || R[i] < lo) lo = R[i];
    if (n_finite == 0 || R[i] > hi) hi = R[i];
    ++n_finite;
  }
  int replaced = n - n_finite;
  if (n_finite == 0 || lo == hi) {
    for (int i = 0; i < n; ++i) Rhat[i] = 0.0;
    return replaced;
  }
  double mu = 0.0;
  for (int i = 0; i < n; ++i) mu += isfinite(R[i]) ? R[i] : lo;
  mu /= (double)n;
  double var = 0.0;
  for (int i = 0; i < n; ++i) {
    double d = (isfinite(R[i]) ? R[i] : lo) - mu;
    var += d * d;
  }
  var /= (double)n;
  double s = sqrt(var);
  for (int i = 0; i < n; ++i)
    Rhat[i] = ((isfinite(R[i]) ? R[i] : lo) - mu) / (s + eps_z);
  return replaced;
}

/*
 * Cosine schedule of sigma over the T generations (§3.1):
 * sigma_t = sigma_T + (sigma_0 - sigma_T) (1 + cos(pi t / T)) / 2, t = 0..T.
 * t is clamped to [0, T]; T <= 0 gives sigma_0.
 */
double oracle_sigma_cosine(double sigma0, double sigmaT, int t, int T) {
  if (T <= 0) return sigma0;
  if (t < 0) t = 0;
  if (t > T) t = T;
  return sigmaT + (sigma0 - sigmaT) * (1.0 + cos(M_PI * (double)t / (double)T)) / 2.0;
}

/*
 * Update coefficients for theta += sum_i c_i eps_i.
 *   mode 0 (paper, §3 and App. D.6):   c_i = alpha * Rhat_i / G
 *   mode 1 (canonical, App. C.1):      c_i = alpha * Rhat_i / (G * sigma)
 * G = n. Computed in double, rounded once to float.
 */
int oracle_update_coeffs(const double* Rhat, int n, double alpha, double sigma,
                         int mode, float* coeffs) {
  if (n < 1 || (mode != 0 && mode != 1)) return -1;
  double denom = (double)n * (mode == 1 ? sigma : 1.0);
  for (int i = 0; i < n; ++i) coeffs[i] = (float)(alpha * Rhat[i] / denom);
  return 0;
}

/*
 * Antithetic pairs: member (i,+) uses +eps_i and member (i,-) uses -eps_i, so
 * the two terms of the update share one noise vector and fold into
 * c_i = alpha * (Rhat_i^+ - Rhat_i^-) / (G * s), with G = 2 * npairs members and
 * s = 1 (mode 0) or sigma (mode 1).
 */
int oracle_fold_antithetic(const double* Rhat_pos, const double* Rhat_neg,
                           int npairs, double alpha, double sigma, int mode,
                           float* coeffs) {
  if (npairs < 1 || (mode != 0 && mode != 1)) return -1;
  double denom = 2.0 * (double)npairs * (mode == 1 ? sigma : 1.0);
  for (int i = 0; i < npairs; ++i)
    coeffs[i] = (float)(alpha * (Rhat_pos[i] - Rhat_neg[i]) / denom);
  return 0;
}

/* Quadratic objective f(theta) = -||theta - theta_star||^2, summed in double. */
double oracle_quadratic_reward(const float* theta, const float* theta_star,
                               uint64_t n) {
  double acc = 0.0;
  for (uint64_t k = 0; k < n; ++k) {
    double d = (double)theta[k] - (double)theta_star[k];
    acc += d * d;
  }
  return -acc;
}
