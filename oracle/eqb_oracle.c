/*
 * eqb_oracle.c -- plain, slow, single-threaded CPU oracle for the EQB + LEI
 * routing-balance path of "Exact Quantile Balancing and Load-Error Injection
 * for Mixture-of-Experts" (arXiv 2609.28053).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  The CUDA product path
 * never calls it, links it or shares code with it.
 *
 * Every function writes out the paper's definition directly:
 *   routing      Sec. 2, Eq. (1) and the QB paragraph: I_t = TopK(z_t + b),
 *                tau_t = (K+1)st largest entry of z_t + b, loads f_e(B).
 *   quantile     Eq. (2): the K/E quantile of the margins tau_t - z_{t,e},
 *                i.e. the r-th smallest (r = TK/E) -- found by a FULL SORT
 *                of each expert's margins (qsort), not by radix selection.
 *   histograms   Algorithm 1, steps 1 and 4 (plain counting loops).
 *   selection    Algorithm 1, steps 3, 5 and 6 (prefix sums, first index
 *                reaching the rank).
 *   bias update  Eq. (2) centering b = b_hat - mean(b_hat).
 *   LEI          Sec. 4, Eq. (LEI) and Eq. (norm).
 *   router       Sec. 2: z_t = W_r x_t, the dot products in fp64.
 *   MaxVio       Sec. 5 (Metrics) and App. E (balance metrics):
 *                max_e [f_e(B) / fbar(B) - 1], global and local.
 *   GShard STE   App. D, Eq. (gshard-grad): the gradient of the GShard
 *                auxiliary loss (Sec. 2) with respect to the router scores.
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   - scores s = fp32(z) + b in fp32 round-to-nearest-even; tau is fp32;
 *   - margin m = bf16_rne(tau - fp32(z)), the subtraction in fp32;
 *   - top-K ties go to the lower expert index; the top-K list is ordered by
 *     score descending, then index ascending;
 *   - r = ceil(T*K/E) (the paper assumes TK/E is an integer);
 *   - kappa maps the bf16 bit pattern x to the 16-bit key
 *       x & 0x8000 ? ~x & 0xffff : x | 0x8000
 *     (so -0 sorts just below +0); a zero quantile is returned as +0;
 *   - margins must be finite with |m| < 2^127: the high bytes 0x00 and 0xff
 *     of kappa hold |m| >= 2^127 and the non-finite patterns alike, so the
 *     coarse pass cannot tell them apart; the quantile and the coarse
 *     histogram refuse margins there (ORACLE_ERR_NONFINITE);
 *   - the centering mean is an fp64 sum in ascending expert order, divided
 *     by E; b_e = (float)((double)b_hat_e - mean);
 *   - LEI adds eta * rho~_e to every (t, e) of the local batch (selected or
 *     not), one shared scale per microbatch, c <= 0 meaning unnormalised;
 *     the injected term and the sum are formed in fp64 and rounded to fp32
 *     once;
 *   - MaxVio in fp64 with fbar = K * |B| / E; Local MaxVio is the plain mean
 *     over the non-empty microbatches (an empty one has no fbar), summed in
 *     ascending microbatch order;
 *   - GShard: the router scores are s = sigmoid(fp32(z)) of the unbiased
 *     logits (Sec. 2), the batch of P^G is the local microbatch, and the
 *     injected term is alpha times the gradient of sum_e F_e P^G_e (the
 *     auxiliary loss), formed in fp64 and added to g with one rounding.
 *
 * Compile with -ffp-contract=off and without -ffast-math.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG 1
#define ORACLE_ERR_NONFINITE 4
#define ORACLE_ERR_NOMEM 5

/* ---- scalar helpers --------------------------------------------------- */

static float bf16_bits_to_f32(uint16_t x) {
  uint32_t u = (uint32_t)x << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

/* Round an fp32 value to bf16, round-to-nearest-even, keeping subnormals.
 * The integer form: add 0x7fff plus the lsb of the kept part, then truncate.
 * NaN is returned as the quiet NaN with the input's sign. */
uint16_t oracle_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu) != 0u)
    return (uint16_t)((u >> 16) | 0x0040u);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7fffu + lsb;
  return (uint16_t)(u >> 16);
}

float oracle_bf16_to_f32(uint16_t x) { return bf16_bits_to_f32(x); }

/* Order-preserving 16-bit key of a bf16 bit pattern (Algorithm 1's kappa). */
uint16_t oracle_kappa(uint16_t x) {
  if (x & 0x8000u) return (uint16_t)(~x & 0xffffu);
  return (uint16_t)(x | 0x8000u);
}

uint16_t oracle_kappa_inv(uint16_t k) {
  if (k & 0x8000u) return (uint16_t)(k & 0x7fffu);
  return (uint16_t)(~k & 0xffffu);
}

static int f32_is_finite(float f) { return isfinite(f) ? 1 : 0; }

int64_t oracle_target_rank(int64_t T, int32_t E, int32_t K) {
  /* r = TK/E, rounded up when TK/E is not an integer (inverse-CDF
   * quantile min{x : F(x) >= K/E}). */
  if (T < 0 || E <= 0 || K <= 0) return -1;
  int64_t num = T * (int64_t)K;
  return (num + E - 1) / E;
}

static int check_offsets(const int64_t *off, int32_t M, int64_t T) {
  if (M < 1 || off == NULL) return 0;
  if (off[0] != 0 || off[M] != T) return 0;
  for (int32_t l = 0; l < M; ++l)
    if (off[l + 1] < off[l]) return 0;
  return 1;
}

/* ---- routing: Sec. 2 ---------------------------------------------------- */

typedef struct {
  float s;
  int32_t e;
} scored_t;

/* Descending score, ties to the lower expert index. */
static int cmp_scored(const void *pa, const void *pb) {
  const scored_t *a = (const scored_t *)pa, *b = (const scored_t *)pb;
  if (a->s > b->s) return -1;
  if (a->s < b->s) return 1;
  return (a->e < b->e) ? -1 : (a->e > b->e) ? 1 : 0;
}

/* For every token t (all T, or only the rows listed in `rows`):
 *   s_e = fp32(z_{t,e}) + b_e; sort (s_e, e) by s descending, e ascending;
 *   idx[t, 0..K-1] = the first K experts; tau[t] = s of the (K+1)-th.
 * loads[l, e] (overwritten, only when rows == NULL) counts the tokens of
 * microbatch l = [off[l], off[l+1]) whose top-K set contains e.
 * With rows != NULL, idx and tau are indexed by position in `rows`. */
int oracle_route(const uint16_t *z, const float *b, int64_t T, int32_t E,
                 int32_t K, const int64_t *off, int32_t M, const int64_t *rows,
                 int64_t n_rows, int32_t *idx, float *tau, int32_t *loads) {
  if (T < 0 || E < 2 || K < 1 || K >= E || z == NULL || b == NULL)
    return ORACLE_ERR_ARG;
  for (int32_t e = 0; e < E; ++e)
    if (!f32_is_finite(b[e])) return ORACLE_ERR_NONFINITE;
  int64_t n = rows ? n_rows : T;
  if (rows == NULL && loads != NULL) {
    if (!check_offsets(off, M, T)) return ORACLE_ERR_ARG;
    memset(loads, 0, sizeof(int32_t) * (size_t)M * (size_t)E);
  }
  scored_t *buf = (scored_t *)malloc(sizeof(scored_t) * (size_t)E);
  if (!buf) return ORACLE_ERR_NOMEM;
  int32_t l = 0;
  for (int64_t i = 0; i < n; ++i) {
    int64_t t = rows ? rows[i] : i;
    if (t < 0 || t >= T) { free(buf); return ORACLE_ERR_ARG; }
    for (int32_t e = 0; e < E; ++e) {
      float zf = bf16_bits_to_f32(z[t * E + e]);
      if (!f32_is_finite(zf)) { free(buf); return ORACLE_ERR_NONFINITE; }
      buf[e].s = zf + b[e];
      buf[e].e = e;
      if (!f32_is_finite(buf[e].s)) { free(buf); return ORACLE_ERR_NONFINITE; }
    }
    qsort(buf, (size_t)E, sizeof(scored_t), cmp_scored);
    if (idx)
      for (int32_t k = 0; k < K; ++k) idx[i * K + k] = buf[k].e;
    if (tau) tau[i] = buf[K].s;
    if (rows == NULL && loads != NULL) {
      while (t >= off[l + 1]) ++l; /* empty microbatches are skipped */
      for (int32_t k = 0; k < K; ++k) loads[(int64_t)l * E + buf[k].e] += 1;
    }
  }
  free(buf);
  return ORACLE_OK;
}

/* A margin the method accepts: finite with |m| < 2^127, i.e. a bf16 pattern
 * whose magnitude bits are below 0x7f00 (kappa high byte 0x01..0xfe). */
static int margin_in_range(uint16_t m) { return (m & 0x7fffu) < 0x7f00u; }

/* ---- margins and the exact quantile: Eq. (2) ---------------------------- */

/* m_{t,e} = bf16_rne(tau_t - fp32(z_{t,e})) for one expert e, all t. */
int oracle_margins(const uint16_t *z, const float *tau, int64_t T, int32_t E,
                   int32_t e, uint16_t *m) {
  if (T < 0 || E < 1 || e < 0 || e >= E) return ORACLE_ERR_ARG;
  for (int64_t t = 0; t < T; ++t) {
    float d = tau[t] - bf16_bits_to_f32(z[t * E + e]);
    m[t] = oracle_f32_to_bf16(d);
  }
  return ORACLE_OK;
}

static int cmp_bf16_value(const void *pa, const void *pb) {
  float a = bf16_bits_to_f32(*(const uint16_t *)pa);
  float b = bf16_bits_to_f32(*(const uint16_t *)pb);
  return (a < b) ? -1 : (a > b) ? 1 : 0;
}

/* b_hat_e = the r-th smallest margin of expert e (1-based r), found by
 * sorting all T margins by value.  A zero result is returned as +0. */
int oracle_quantile(const uint16_t *z, const float *tau, int64_t T, int32_t E,
                    int64_t r, const int32_t *experts, int32_t n_experts,
                    uint16_t *qhat) {
  if (T < 1 || r < 1 || r > T || E < 1) return ORACLE_ERR_ARG;
  uint16_t *m = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)T);
  if (!m) return ORACLE_ERR_NOMEM;
  for (int32_t i = 0; i < n_experts; ++i) {
    int32_t e = experts ? experts[i] : i;
    if (e < 0 || e >= E) { free(m); return ORACLE_ERR_ARG; }
    oracle_margins(z, tau, T, E, e, m);
    for (int64_t t = 0; t < T; ++t)
      if (!margin_in_range(m[t])) { free(m); return ORACLE_ERR_NONFINITE; }
    qsort(m, (size_t)T, sizeof(uint16_t), cmp_bf16_value);
    uint16_t q = m[r - 1];
    if (q == 0x8000u) q = 0; /* zero is returned as +0 */
    qhat[i] = q;
  }
  free(m);
  return ORACLE_OK;
}

/* ---- Algorithm 1 counts and selections ---------------------------------- */

/* Step 1: H[e][u] = #{t : high byte of kappa(m_{t,e}) == u}.  Overwrites H
 * [E,256] for tokens [t0, t1). */
int oracle_hist_hi(const uint16_t *z, const float *tau, int64_t t0, int64_t t1,
                   int32_t E, int32_t *H) {
  if (t0 < 0 || t1 < t0 || E < 1) return ORACLE_ERR_ARG;
  memset(H, 0, sizeof(int32_t) * (size_t)E * 256u);
  for (int64_t t = t0; t < t1; ++t)
    for (int32_t e = 0; e < E; ++e) {
      uint16_t m = oracle_f32_to_bf16(tau[t] - bf16_bits_to_f32(z[t * E + e]));
      if (!margin_in_range(m)) return ORACLE_ERR_NONFINITE;
      uint16_t k = oracle_kappa(m);
      H[(int64_t)e * 256 + (k >> 8)] += 1;
    }
  return ORACLE_OK;
}

/* Step 4: L[e][v] = #{t : kappa(m_{t,e}) == (u_e, v)}.  Overwrites L. */
int oracle_hist_lo(const uint16_t *z, const float *tau, int64_t t0, int64_t t1,
                   int32_t E, const uint8_t *u, int32_t *L) {
  if (t0 < 0 || t1 < t0 || E < 1) return ORACLE_ERR_ARG;
  memset(L, 0, sizeof(int32_t) * (size_t)E * 256u);
  for (int64_t t = t0; t < t1; ++t)
    for (int32_t e = 0; e < E; ++e) {
      uint16_t m = oracle_f32_to_bf16(tau[t] - bf16_bits_to_f32(z[t * E + e]));
      uint16_t k = oracle_kappa(m);
      if ((k >> 8) == u[e]) L[(int64_t)e * 256 + (k & 0xffu)] += 1;
    }
  return ORACLE_OK;
}

/* Step 3: u_e = min{u : sum_{j<=u} H[e][j] >= r};
 *         rho_e = r - sum_{j<u_e} H[e][j]. */
int oracle_select_hi(const int32_t *H, int32_t E, int64_t r, uint8_t *u,
                     int32_t *rho) {
  if (E < 1 || r < 1) return ORACLE_ERR_ARG;
  for (int32_t e = 0; e < E; ++e) {
    int64_t below = 0;
    int found = 0;
    for (int32_t j = 0; j < 256; ++j) {
      int64_t c = H[(int64_t)e * 256 + j];
      if (below + c >= r) {
        u[e] = (uint8_t)j;
        rho[e] = (int32_t)(r - below);
        found = 1;
        break;
      }
      below += c;
    }
    if (!found) return ORACLE_ERR_ARG; /* fewer than r margins counted */
  }
  return ORACLE_OK;
}

/* Steps 5-6: v_e = min{v : sum_{j<=v} L[e][j] >= rho_e};
 *            b_hat_e = kappa^{-1}(u_e, v_e), zero returned as +0. */
int oracle_select_lo(const int32_t *L, int32_t E, const uint8_t *u,
                     const int32_t *rho, uint16_t *qhat) {
  if (E < 1) return ORACLE_ERR_ARG;
  for (int32_t e = 0; e < E; ++e) {
    int64_t below = 0;
    int found = 0;
    for (int32_t j = 0; j < 256; ++j) {
      below += L[(int64_t)e * 256 + j];
      if (below >= rho[e]) {
        uint16_t q = oracle_kappa_inv((uint16_t)(((uint16_t)u[e] << 8) | (uint16_t)j));
        if (q == 0x8000u) q = 0;
        qhat[e] = q;
        found = 1;
        break;
      }
    }
    if (!found) return ORACLE_ERR_ARG;
  }
  return ORACLE_OK;
}

/* ---- Eq. (2) centering -------------------------------------------------- */

int oracle_bias_update(const uint16_t *qhat, int32_t E, float *b_next) {
  if (E < 1) return ORACLE_ERR_ARG;
  double sum = 0.0;
  for (int32_t e = 0; e < E; ++e) sum += (double)bf16_bits_to_f32(qhat[e]);
  double mean = sum / (double)E;
  for (int32_t e = 0; e < E; ++e)
    b_next[e] = (float)((double)bf16_bits_to_f32(qhat[e]) - mean);
  return ORACLE_OK;
}

/* ---- LEI: Sec. 4, Eq. (LEI) and Eq. (norm) ------------------------------ */

/* Per microbatch l with n_l tokens and loads f_{l,e}:
 *   fbar = K n_l / E;  rho_e = f_e / fbar - 1;
 *   c > 0:  xi = max_e |rho_e| / c,  sigma = tanh(xi)/xi  (1 at xi = 0);
 *   c <= 0: sigma = 1 (unnormalised LEI);
 *   a_{l,e} = eta * sigma * rho_e;
 *   g_out[t, e] = fp32(g[t, e] + a_{l,e}) for every t in the microbatch.
 * a_out [M,E] (optional) receives the fp64 coefficients.  Empty microbatches
 * get a = 0. */
int oracle_lei(const float *g, const int32_t *loads, const int64_t *off,
               int32_t M, int64_t T, int32_t E, int32_t K, float eta, float c,
               float *g_out, double *a_out) {
  if (T < 0 || E < 1 || K < 1 || !check_offsets(off, M, T)) return ORACLE_ERR_ARG;
  double *a = (double *)malloc(sizeof(double) * (size_t)E);
  if (!a) return ORACLE_ERR_NOMEM;
  for (int32_t l = 0; l < M; ++l) {
    int64_t n = off[l + 1] - off[l];
    if (n == 0) {
      for (int32_t e = 0; e < E; ++e) a[e] = 0.0;
    } else {
      double fbar = (double)K * (double)n / (double)E;
      double rmax = 0.0;
      for (int32_t e = 0; e < E; ++e) {
        a[e] = (double)loads[(int64_t)l * E + e] / fbar - 1.0;
        if (fabs(a[e]) > rmax) rmax = fabs(a[e]);
      }
      double sigma = 1.0;
      if (c > 0.0f) {
        double xi = rmax / (double)c;
        sigma = (xi == 0.0) ? 1.0 : tanh(xi) / xi;
      }
      for (int32_t e = 0; e < E; ++e) a[e] = (double)eta * sigma * a[e];
    }
    if (a_out)
      for (int32_t e = 0; e < E; ++e) a_out[(int64_t)l * E + e] = a[e];
    if (g != NULL && g_out != NULL)
      for (int64_t t = off[l]; t < off[l + 1]; ++t)
        for (int32_t e = 0; e < E; ++e)
          g_out[t * E + e] = (float)((double)g[t * E + e] + a[e]);
  }
  free(a);
  return ORACLE_OK;
}

/* ---- router projection: Sec. 2, z_t = W_r x_t -------------------------- */

/* For each listed row t: out[i, e] = sum_k x[t, k] * W[e, k] in fp64 (each
 * product of two bf16 values is exact in fp64) and abs_out[i, e] =
 * sum_k |x[t, k] * W[e, k]| (the scale of the accumulation error). */
int oracle_router_logits(const uint16_t *x, const uint16_t *W, int64_t T, int32_t d, int32_t E,
                         const int64_t *rows, int64_t n_rows, double *out, double *abs_out) {
  if (T < 0 || d < 1 || E < 1) return ORACLE_ERR_ARG;
  for (int64_t i = 0; i < n_rows; ++i) {
    int64_t t = rows[i];
    if (t < 0 || t >= T) return ORACLE_ERR_ARG;
    for (int32_t e = 0; e < E; ++e) {
      double acc = 0.0, acc_abs = 0.0;
      for (int32_t k = 0; k < d; ++k) {
        double p = (double)bf16_bits_to_f32(x[t * d + k]) * (double)bf16_bits_to_f32(W[(int64_t)e * d + k]);
        acc += p;
        acc_abs += fabs(p);
      }
      out[i * E + e] = acc;
      if (abs_out) abs_out[i * E + e] = acc_abs;
    }
  }
  return ORACLE_OK;
}

/* ---- balance metric: Sec. 5 (Metrics), App. E --------------------------- */

/* MaxVio(B) = max_e [ f_e(B) / fbar(B) - 1 ], fbar(B) = K |B| / E, in fp64.
 *   global   loads summed over all microbatches, |B| = T = off[M];
 *   local    MaxVio of every non-empty microbatch l (|B| = off[l+1] - off[l])
 *            and their plain mean, summed in ascending l; per_mb (optional,
 *            [M]) receives each microbatch's value (0 for an empty one).
 * Returns ORACLE_ERR_ARG when every microbatch is empty. */
int oracle_maxvio(const int32_t *loads, const int64_t *off, int32_t M, int32_t E, int32_t K,
                  double *global, double *local, double *per_mb) {
  if (E < 1 || K < 1 || M < 1 || off == NULL || off[0] != 0) return ORACLE_ERR_ARG;
  int64_t T = off[M];
  if (T < 1 || !check_offsets(off, M, T)) return ORACLE_ERR_ARG;
  double sum = 0.0;
  int32_t count = 0;
  for (int32_t l = 0; l < M; ++l) {
    int64_t n = off[l + 1] - off[l];
    double v = 0.0;
    if (n > 0) {
      const double fbar_l = (double)K * (double)n / (double)E;
      v = -INFINITY;
      for (int32_t e = 0; e < E; ++e) {
        double x = (double)loads[(int64_t)l * E + e] / fbar_l - 1.0;
        if (x > v) v = x;
      }
      sum += v;
      ++count;
    }
    if (per_mb) per_mb[l] = v;
  }
  double fbar = (double)K * (double)T / (double)E;
  double g = -INFINITY;
  for (int32_t e = 0; e < E; ++e) {
    int64_t f = 0;
    for (int32_t l = 0; l < M; ++l) f += loads[(int64_t)l * E + e];
    double x = (double)f / fbar - 1.0;
    if (x > g) g = x;
  }
  *global = g;
  *local = sum / (double)count;
  return ORACLE_OK;
}

/* ---- GShard auxiliary-loss gradient: App. D, Eq. (gshard-grad) ---------- */

/* For microbatch l with n tokens and loads f_e:  F_e = f_e / (K n),
 * R_e = F_e - 1/E; for each of its tokens t, with s_e = sigmoid(z_{t,e}),
 * d_t = sum_e s_e and p_e = s_e / d_t,
 *   g_out[t, j] = fp32( g[t, j] + alpha / (n d_t) * (R_j - sum_e p_e R_e) ),
 * all in fp64.  Empty microbatches have no tokens. */
int oracle_gshard(const float *g, const uint16_t *z, const int32_t *loads, const int64_t *off,
                  int32_t M, int64_t T, int32_t E, int32_t K, float alpha, float *g_out) {
  if (T < 0 || E < 1 || K < 1 || !check_offsets(off, M, T)) return ORACLE_ERR_ARG;
  double *R = (double *)malloc(sizeof(double) * (size_t)E);
  double *s = (double *)malloc(sizeof(double) * (size_t)E);
  if (!R || !s) {
    free(R);
    free(s);
    return ORACLE_ERR_NOMEM;
  }
  for (int32_t l = 0; l < M; ++l) {
    const int64_t n = off[l + 1] - off[l];
    if (n == 0) continue;
    for (int32_t e = 0; e < E; ++e)
      R[e] = (double)loads[(int64_t)l * E + e] / ((double)K * (double)n) - 1.0 / (double)E;
    for (int64_t t = off[l]; t < off[l + 1]; ++t) {
      double d = 0.0;
      for (int32_t e = 0; e < E; ++e) {
        s[e] = 1.0 / (1.0 + exp(-(double)bf16_bits_to_f32(z[t * E + e])));
        d += s[e];
      }
      double m = 0.0;
      for (int32_t e = 0; e < E; ++e) m += (s[e] / d) * R[e];
      const double scale = (double)alpha / ((double)n * d);
      for (int32_t j = 0; j < E; ++j)
        g_out[t * E + j] = (float)((double)g[t * E + j] + scale * (R[j] - m));
    }
  }
  free(R);
  free(s);
  return ORACLE_OK;
}
