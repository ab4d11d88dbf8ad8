/*
 * CPU oracle for the MOBO candidate-scoring step of BOute (arXiv 2602.10729).
 * TEST INFRASTRUCTURE ONLY: see boute_oracle.h. Plain fp64 C, no BLAS, no
 * blocking or reordering beyond the textbook definitions cited per function.
 */
#include "boute_oracle.h"

#define _GNU_SOURCE
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

int bo_default_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

static int nthreads_or_default(int nthreads) {
  return nthreads > 0 ? nthreads : bo_default_threads();
}

/* ---- Sec. 6: Standardize outcome transform ------------------------------ */
int bo_standardize(const double *Y, int n, int m, double *Ys) {
  if (n < 0 || m < 1 || (n > 0 && (!Y || !Ys))) return 1;
  for (int t = 0; t < m; ++t) {
    double mean = 0.0;
    for (int i = 0; i < n; ++i) mean += Y[(long)i * m + t];
    mean = n > 0 ? mean / n : 0.0;
    double ss = 0.0;
    for (int i = 0; i < n; ++i) {
      double z = Y[(long)i * m + t] - mean;
      ss += z * z;
    }
    double sd = n > 1 ? sqrt(ss / (n - 1)) : 1.0;
    if (!(sd >= 1e-8)) sd = 1.0;
    for (int i = 0; i < n; ++i) Ys[(long)i * m + t] = (Y[(long)i * m + t] - mean) / sd;
  }
  return 0;
}

/* ---- Sec. 6 (i): ARD Matern-5/2 with ScaleKernel ------------------------ */
double bo_matern52(const double *a, const double *b, int d, const double *ls, double s2) {
  double r2 = 0.0;
  for (int t = 0; t < d; ++t) {
    double z = (a[t] - b[t]) / ls[t];
    r2 += z * z;
  }
  double r = sqrt(r2);
  double sr = sqrt(5.0) * r;
  return s2 * (1.0 + sr + 5.0 * r2 / 3.0) * exp(-sr);
}

/* ---- Sec. 6 (ii): ARD Matern-3/2 with ScaleKernel ------------------------ */
double bo_matern32(const double *a, const double *b, int d, const double *ls, double s2) {
  double r2 = 0.0;
  for (int t = 0; t < d; ++t) {
    double z = (a[t] - b[t]) / ls[t];
    r2 += z * z;
  }
  double sr = sqrt(3.0) * sqrt(r2);
  return s2 * (1.0 + sr) * exp(-sr);
}

/* ---- Sec. 5.2 S1-S3 / S5: preference weight of a deployment --------------- */
double bo_pref_weight(const double *c, int dc, double beta, const double *pref) {
  double e = 0.0;
  for (int k = 0; k < dc; ++k) e += pref[k] * c[k];
  return exp(beta * e);
}

/* ---- Sec. 5.2 "Additive kernels" and Sec. 6 (i)-(iv): the GP's kernel ------ */
double bo_kernel(const double *a, const double *b, int d, const double *ls, double s2,
                 int dtau, const double *kc) {
  if (!kc) return bo_matern52(a, b, d, ls, s2);
  const int dc = d - dtau;
  /* the base kernels, unscaled: k_tau over the routing features, k_c over the
   * deployment features (ProductKernel(k_tau, k_c) reuses both) */
  double ktau = bo_matern52(a, b, dtau, ls, 1.0);
  double kcd = bo_matern32(a + dtau, b + dtau, dc, ls + dtau, 1.0);
  double wa = bo_pref_weight(a + dtau, dc, kc[2], kc + 3);
  double wb = bo_pref_weight(b + dtau, dc, kc[2], kc + 3);
  return s2 * ktau + kc[0] * wa * wb * kcd + kc[1] * ktau * kcd;
}

/* ---- Sec. 5.2 S4: outcome transforms applied before Standardize ----------- */
int bo_outcome_transform(const double *Y, int n, int m, const int *codes, double *Yt) {
  if (n < 0 || m < 1 || (n > 0 && (!Y || !Yt))) return 1;
  for (int i = 0; i < n; ++i)
    for (int t = 0; t < m; ++t) {
      double y = Y[(long)i * m + t];
      int c = codes ? codes[t] : 0;
      double v = y;
      if ((c & 3) == 1) v = log(y);                  /* latency: log */
      else if ((c & 3) == 2) v = log(y / (1.0 - y)); /* quality: logit */
      if (c & 4) v = -v;                             /* a maximised outcome, minimised */
      Yt[(long)i * m + t] = v;
    }
  return 0;
}

/* ---- Sec. 5.2 (i) / Sec. 6: exact GP fit --------------------------------- */
int bo_gp_fit(const double *X, const double *y, int n, int d, const double *ls,
              double s2, double noise, double *L, double *alpha) {
  return bo_gp_fit_k(X, y, n, d, ls, s2, noise, d, NULL, L, alpha);
}

int bo_gp_fit_k(const double *X, const double *y, int n, int d, const double *ls, double s2,
                double noise, int dtau, const double *kc, double *L, double *alpha) {
  if (n < 1 || d < 1 || !X || !y || !ls || !L || !alpha) return 1;
  if (kc && (dtau < 0 || dtau > d)) return 1;
  /* K = k(X, X) + noise I, lower triangle written straight into L */
  for (int i = 0; i < n; ++i)
    for (int j = 0; j < n; ++j)
      L[(long)i * n + j] =
          j <= i ? bo_kernel(X + (long)i * d, X + (long)j * d, d, ls, s2, dtau, kc) +
                       (i == j ? noise : 0.0)
                 : 0.0;
  /* Cholesky-Banachiewicz, row by row, in place */
  for (int i = 0; i < n; ++i) {
    for (int j = 0; j <= i; ++j) {
      double s = L[(long)i * n + j];
      for (int k = 0; k < j; ++k) s -= L[(long)i * n + k] * L[(long)j * n + k];
      if (i == j) {
        if (!(s > 0.0)) return 2;
        L[(long)i * n + i] = sqrt(s);
      } else {
        L[(long)i * n + j] = s / L[(long)j * n + j];
      }
    }
  }
  /* alpha = L^-T (L^-1 y) */
  for (int i = 0; i < n; ++i) {
    double s = y[i];
    for (int k = 0; k < i; ++k) s -= L[(long)i * n + k] * alpha[k];
    alpha[i] = s / L[(long)i * n + i];
  }
  for (int i = n - 1; i >= 0; --i) {
    double s = alpha[i];
    for (int k = i + 1; k < n; ++k) s -= L[(long)k * n + i] * alpha[k];
    alpha[i] = s / L[(long)i * n + i];
  }
  return 0;
}

void bo_gp_posterior(const double *X, int n, int d, const double *ls, double s2,
                     const double *L, const double *alpha, const float *Xc,
                     long long N, double *mean, double *var, int nthreads) {
  bo_gp_posterior_k(X, n, d, ls, s2, d, NULL, L, alpha, Xc, N, mean, var, nthreads);
}

void bo_gp_posterior_k(const double *X, int n, int d, const double *ls, double s2, int dtau,
                       const double *kc, const double *L, const double *alpha, const float *Xc,
                       long long N, double *mean, double *var, int nthreads) {
  int nt = nthreads_or_default(nthreads);
  /* prior variance k(x, x): s2 for the Matern-5/2 kernel; for the composite
   * kernel it depends on x through the preference weight */
#pragma omp parallel num_threads(nt)
  {
    double *kv = (double *)malloc(sizeof(double) * (size_t)(2 * n + d));
    double *v = kv + n, *xc = kv + 2 * n;
#pragma omp for schedule(static)
    for (long long c = 0; c < N; ++c) {
      for (int t = 0; t < d; ++t) xc[t] = (double)Xc[c * d + t];
      double mu = 0.0;
      for (int j = 0; j < n; ++j) {
        kv[j] = bo_kernel(xc, X + (long)j * d, d, ls, s2, dtau, kc);
        mu += kv[j] * alpha[j];
      }
      double vv = 0.0;
      for (int i = 0; i < n; ++i) { /* v = L^-1 k* */
        double s = kv[i];
        for (int j = 0; j < i; ++j) s -= L[(long)i * n + j] * v[j];
        v[i] = s / L[(long)i * n + i];
        vv += v[i] * v[i];
      }
      double s2v = bo_kernel(xc, xc, d, ls, s2, dtau, kc) - vv;
      mean[c] = mu;
      var[c] = s2v > 0.0 ? s2v : 0.0;
    }
    free(kv);
  }
}

/* ---- Sec. 6: hyperparameters learned by maximising the marginal likelihood */
double bo_gp_mll(const double *X, const double *y, int n, int d, const double *ls, double s2,
                 double noise, double *grad) {
  double *L = (double *)malloc(sizeof(double) * ((size_t)n * n * 2 + 2 * (size_t)n));
  double *Ki = L + (size_t)n * n, *alpha = Ki + (size_t)n * n, *col = alpha + n;
  double mll = NAN;
  if (bo_gp_fit(X, y, n, d, ls, s2, noise, L, alpha) != 0) goto done;
  /* log p(y) = -1/2 y^T alpha - sum_i log L_ii - n/2 log(2 pi) */
  mll = -0.5 * (double)n * log(2.0 * M_PI);
  for (int i = 0; i < n; ++i) mll += -0.5 * y[i] * alpha[i] - log(L[(long)i * n + i]);
  if (grad) {
    /* K^-1 column by column: solve L L^T x = e_j */
    for (int j = 0; j < n; ++j) {
      for (int i = 0; i < n; ++i) {
        double s = i == j ? 1.0 : 0.0;
        for (int k = 0; k < i; ++k) s -= L[(long)i * n + k] * col[k];
        col[i] = s / L[(long)i * n + i];
      }
      for (int i = n - 1; i >= 0; --i) {
        double s = col[i];
        for (int k = i + 1; k < n; ++k) s -= L[(long)k * n + i] * col[k];
        col[i] = s / L[(long)i * n + i];
      }
      for (int i = 0; i < n; ++i) Ki[(long)i * n + j] = col[i];
    }
    /* d log p / d theta = 1/2 tr((alpha alpha^T - K^-1) dK/dtheta), theta the
     * log-parameters: dK/dlog s2 = s2 M52; dK/dlog noise = noise I;
     * dK_ij/dlog l_t = s2 (5/3) (1 + sqrt5 r) exp(-sqrt5 r) (dx_t / l_t)^2 */
    for (int q = 0; q < d + 2; ++q) grad[q] = 0.0;
    for (int i = 0; i < n; ++i)
      for (int j = 0; j < n; ++j) {
        const double Q = alpha[i] * alpha[j] - Ki[(long)i * n + j];
        const double *xi = X + (long)i * d, *xj = X + (long)j * d;
        double r2 = 0.0;
        for (int t = 0; t < d; ++t) {
          double z = (xi[t] - xj[t]) / ls[t];
          r2 += z * z;
        }
        const double r = sqrt(r2), e = exp(-sqrt(5.0) * r);
        const double f = s2 * (5.0 / 3.0) * (1.0 + sqrt(5.0) * r) * e;
        for (int t = 0; t < d; ++t) {
          double z = (xi[t] - xj[t]) / ls[t];
          grad[t] += 0.5 * Q * f * z * z;
        }
        grad[d] += 0.5 * Q * s2 * (1.0 + sqrt(5.0) * r + 5.0 * r2 / 3.0) * e;
        if (i == j) grad[d + 1] += 0.5 * Q * noise;
      }
  }
done:
  free(L);
  return mll;
}

/* The composite kernel's log marginal likelihood and its gradient with respect
 * to theta = (log l_1..log l_d, log s2, log noise, log s2_c, log s2_x, beta).
 * Per entry, with the routing distance r_t, the deployment distance r_c,
 * e5 = exp(-sqrt5 r_t), e3 = exp(-sqrt3 r_c) and ww = w_i w_j:
 *   dK/dlog l_q (routing)    = (5/3)(1 + sqrt5 r_t) e5 z_q^2 (s2 + s2_x k32)
 *   dK/dlog l_q (deployment) = 3 e3 z_q^2 (s2_c ww + s2_x k52)
 *   dK/dlog s2 = s2 k52, dK/dlog s2_c = s2_c ww k32, dK/dlog s2_x = s2_x k52 k32,
 *   dK/dbeta = s2_c ww k32 (<s, c_i> + <s, c_j>), dK/dlog noise = noise I. */
double bo_gp_mll_k(const double *X, const double *y, int n, int d, const double *ls, double s2,
                   double noise, int dtau, const double *kc, double *grad) {
  double *L = (double *)malloc(sizeof(double) * ((size_t)n * n * 2 + 3 * (size_t)n));
  double *Ki = L + (size_t)n * n, *alpha = Ki + (size_t)n * n, *col = alpha + n, *pc = col + n;
  double mll = NAN;
  const int dc = d - dtau;
  if (bo_gp_fit_k(X, y, n, d, ls, s2, noise, dtau, kc, L, alpha) != 0) goto done;
  mll = -0.5 * (double)n * log(2.0 * M_PI);
  for (int i = 0; i < n; ++i) mll += -0.5 * y[i] * alpha[i] - log(L[(long)i * n + i]);
  if (grad) {
    for (int j = 0; j < n; ++j) {
      for (int i = 0; i < n; ++i) {
        double s = i == j ? 1.0 : 0.0;
        for (int k = 0; k < i; ++k) s -= L[(long)i * n + k] * col[k];
        col[i] = s / L[(long)i * n + i];
      }
      for (int i = n - 1; i >= 0; --i) {
        double s = col[i];
        for (int k = i + 1; k < n; ++k) s -= L[(long)k * n + i] * col[k];
        col[i] = s / L[(long)i * n + i];
      }
      for (int i = 0; i < n; ++i) Ki[(long)i * n + j] = col[i];
    }
    for (int i = 0; i < n; ++i) { /* <s, c_i> */
      double e = 0.0;
      for (int k = 0; k < dc; ++k) e += kc[3 + k] * X[(long)i * d + dtau + k];
      pc[i] = e;
    }
    const double s2c = kc[0], s2x = kc[1], beta = kc[2];
    for (int q = 0; q < d + 5; ++q) grad[q] = 0.0;
    for (int i = 0; i < n; ++i)
      for (int j = 0; j < n; ++j) {
        const double Q = 0.5 * (alpha[i] * alpha[j] - Ki[(long)i * n + j]);
        const double *xi = X + (long)i * d, *xj = X + (long)j * d;
        double rt2 = 0.0, rc2 = 0.0;
        for (int t = 0; t < d; ++t) {
          double z = (xi[t] - xj[t]) / ls[t];
          if (t < dtau) rt2 += z * z;
          else rc2 += z * z;
        }
        const double rt = sqrt(rt2), rc = sqrt(rc2);
        const double e5 = exp(-sqrt(5.0) * rt), e3 = exp(-sqrt(3.0) * rc);
        const double k52 = (1.0 + sqrt(5.0) * rt + 5.0 * rt2 / 3.0) * e5;
        const double k32 = (1.0 + sqrt(3.0) * rc) * e3;
        const double ww = exp(beta * (pc[i] + pc[j]));
        for (int t = 0; t < d; ++t) {
          double z = (xi[t] - xj[t]) / ls[t];
          if (t < dtau)
            grad[t] += Q * (5.0 / 3.0) * (1.0 + sqrt(5.0) * rt) * e5 * z * z * (s2 + s2x * k32);
          else
            grad[t] += Q * 3.0 * e3 * z * z * (s2c * ww + s2x * k52);
        }
        grad[d] += Q * s2 * k52;
        if (i == j) grad[d + 1] += Q * noise;
        grad[d + 2] += Q * s2c * ww * k32;
        grad[d + 3] += Q * s2x * k52 * k32;
        grad[d + 4] += Q * s2c * ww * k32 * (pc[i] + pc[j]);
      }
  }
done:
  free(L);
  return mll;
}

/* Log-parameter bounds of the learner (theta = log l_1..log l_d, log s2, log noise). */
static double clampd(double v, double lo, double hi) { return v < lo ? lo : (v > hi ? hi : v); }
static void learn_clamp(double *th, int d) {
  for (int t = 0; t < d; ++t) th[t] = clampd(th[t], BO_LOG_LS_MIN, BO_LOG_LS_MAX);
  th[d] = clampd(th[d], BO_LOG_S2_MIN, BO_LOG_S2_MAX);
  th[d + 1] = clampd(th[d + 1], BO_LOG_NOISE_MIN, BO_LOG_NOISE_MAX);
}
/* the composite kernel's extra parameters (log s2_c, log s2_x, beta) */
static void learn_clamp_k(double *th, int d) {
  th[d + 2] = clampd(th[d + 2], BO_LOG_SC_MIN, BO_LOG_SC_MAX);
  th[d + 3] = clampd(th[d + 3], BO_LOG_SC_MIN, BO_LOG_SC_MAX);
  th[d + 4] = clampd(th[d + 4], BO_BETA_MIN, BO_BETA_MAX);
}

static double mll_at(const double *X, const double *y, int n, int d, const double *th,
                     double *grad, double *ls) {
  for (int t = 0; t < d; ++t) ls[t] = exp(th[t]);
  return bo_gp_mll(X, y, n, d, ls, exp(th[d]), exp(th[d + 1]), grad);
}

int bo_gp_learn(const double *X, const double *y, int n, int d, const double *theta0, int R,
                int iters, double lr, double *theta, double *mll, double *grad) {
  if (n < 1 || d < 1 || R < 1 || iters < 0 || !X || !y || !theta0 || !theta || !mll) return 1;
  const int P = d + 2;
  double *buf = (double *)malloc(sizeof(double) * (size_t)(4 * P + d));
  double *g = buf, *m1 = g + P, *m2 = m1 + P, *ls = m2 + P;
  for (int r = 0; r < R; ++r) {
    double *th = theta + (size_t)r * P;
    memcpy(th, theta0 + (size_t)r * P, sizeof(double) * P);
    learn_clamp(th, d);
    for (int q = 0; q < P; ++q) m1[q] = m2[q] = 0.0;
    double b1t = 1.0, b2t = 1.0;
    for (int it = 0; it < iters; ++it) {
      /* Adam ascent on the log marginal likelihood, bias-corrected moments */
      const double v = mll_at(X, y, n, d, th, g, ls);
      if (v != v) break; /* not positive definite: keep the last theta */
      b1t *= BO_ADAM_B1;
      b2t *= BO_ADAM_B2;
      for (int q = 0; q < P; ++q) {
        m1[q] = BO_ADAM_B1 * m1[q] + (1.0 - BO_ADAM_B1) * g[q];
        m2[q] = BO_ADAM_B2 * m2[q] + (1.0 - BO_ADAM_B2) * g[q] * g[q];
        const double mh = m1[q] / (1.0 - b1t), vh = m2[q] / (1.0 - b2t);
        th[q] += lr * mh / (sqrt(vh) + BO_ADAM_EPS);
      }
      learn_clamp(th, d);
    }
    mll[r] = mll_at(X, y, n, d, th, grad ? grad + (size_t)r * P : NULL, ls);
  }
  free(buf);
  return 0;
}

static double mll_at_k(const double *X, const double *y, int n, int d, int dtau,
                       const double *pref, const double *th, double *grad, double *ls,
                       double *kc) {
  for (int t = 0; t < d; ++t) ls[t] = exp(th[t]);
  kc[0] = exp(th[d + 2]);
  kc[1] = exp(th[d + 3]);
  kc[2] = th[d + 4];
  for (int k = 0; k < d - dtau; ++k) kc[3 + k] = pref[k];
  return bo_gp_mll_k(X, y, n, d, ls, exp(th[d]), exp(th[d + 1]), dtau, kc, grad);
}

int bo_gp_learn_k(const double *X, const double *y, int n, int d, int dtau, const double *pref,
                  const double *theta0, int R, int iters, double lr, double *theta, double *mll,
                  double *grad) {
  if (n < 1 || d < 1 || dtau < 0 || dtau > d || R < 1 || iters < 0 || !X || !y || !pref ||
      !theta0 || !theta || !mll)
    return 1;
  const int P = d + 5;
  double *buf = (double *)malloc(sizeof(double) * (size_t)(3 * P + d + 3 + d));
  double *g = buf, *m1 = g + P, *m2 = m1 + P, *ls = m2 + P, *kc = ls + d;
  for (int r = 0; r < R; ++r) {
    double *th = theta + (size_t)r * P;
    memcpy(th, theta0 + (size_t)r * P, sizeof(double) * P);
    learn_clamp(th, d);
    learn_clamp_k(th, d);
    for (int q = 0; q < P; ++q) m1[q] = m2[q] = 0.0;
    double b1t = 1.0, b2t = 1.0;
    for (int it = 0; it < iters; ++it) {
      const double v = mll_at_k(X, y, n, d, dtau, pref, th, g, ls, kc);
      if (v != v) break; /* not positive definite: keep the last theta */
      b1t *= BO_ADAM_B1;
      b2t *= BO_ADAM_B2;
      for (int q = 0; q < P; ++q) {
        m1[q] = BO_ADAM_B1 * m1[q] + (1.0 - BO_ADAM_B1) * g[q];
        m2[q] = BO_ADAM_B2 * m2[q] + (1.0 - BO_ADAM_B2) * g[q] * g[q];
        const double mh = m1[q] / (1.0 - b1t), vh = m2[q] / (1.0 - b2t);
        th[q] += lr * mh / (sqrt(vh) + BO_ADAM_EPS);
      }
      learn_clamp(th, d);
      learn_clamp_k(th, d);
    }
    mll[r] = mll_at_k(X, y, n, d, dtau, pref, th, grad ? grad + (size_t)r * P : NULL, ls, kc);
  }
  free(buf);
  return 0;
}

/* ---- Monte-Carlo base normals from a counter-based generator ------------
 * Philox4x64-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two
 * 64 x 64 -> 128-bit products with a Weyl key schedule; normals by the
 * Box-Muller transform of its 53-bit uniforms. */
static void mulhilo64(unsigned long long a, unsigned long long b, unsigned long long *hi,
                      unsigned long long *lo) {
  const unsigned __int128 p = (unsigned __int128)a * b;
  *hi = (unsigned long long)(p >> 64);
  *lo = (unsigned long long)p;
}

void bo_philox4x64(const unsigned long long ctr[4], const unsigned long long key[2],
                   unsigned long long out[4]) {
  unsigned long long c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3], k0 = key[0],
                     k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    unsigned long long hi0, lo0, hi1, lo1;
    mulhilo64(0xD2E7470EE14C6C93ull, c0, &hi0, &lo0);
    mulhilo64(0xCA5A826395121157ull, c2, &hi1, &lo1);
    const unsigned long long n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
    k0 += 0x9E3779B97F4A7C15ull;
    k1 += 0xBB67AE8584CAA73Bull;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

void bo_base_normals(unsigned long long seed, int B, long long N, int m, int S, float *eps) {
  const unsigned long long key[2] = {seed, 0ull};
  for (int b = 0; b < B; ++b)
    for (long long c = 0; c < N; ++c)
      for (int t = 0; t < m; ++t) {
        float *e = eps + (((size_t)b * N + c) * m + t) * S;
        for (int j = 0; 4 * j < S; ++j) {
          const unsigned long long ctr[4] = {(unsigned long long)j, (unsigned long long)c,
                                             (unsigned long long)b * m + t, 0ull};
          unsigned long long w[4];
          bo_philox4x64(ctr, key, w);
          double u[4];
          for (int q = 0; q < 4; ++q) u[q] = ((double)(w[q] >> 11) + 0.5) * 0x1p-53;
          for (int q = 0; q < 2; ++q) {
            const double rad = sqrt(-2.0 * log(u[2 * q])), ang = 2.0 * M_PI * u[2 * q + 1];
            if (4 * j + 2 * q < S) e[4 * j + 2 * q] = (float)(rad * cos(ang));
            if (4 * j + 2 * q + 1 < S) e[4 * j + 2 * q + 1] = (float)(rad * sin(ang));
          }
        }
      }
}

/* ---- Sec. 5.2: Pareto-optimal set (minimisation) ------------------------- */
static _Thread_local const double *g_sortY;
static _Thread_local int g_sortM;
static int cmp_lex(const void *pa, const void *pb) {
  int a = *(const int *)pa, b = *(const int *)pb;
  for (int t = 0; t < g_sortM; ++t) {
    double ya = g_sortY[(long)a * g_sortM + t], yb = g_sortY[(long)b * g_sortM + t];
    if (ya < yb) return -1;
    if (ya > yb) return 1;
  }
  return (a > b) - (a < b);
}

int bo_pareto_front(const double *Y, int n, int m, const double *ref,
                    unsigned char *mask, int *order) {
  if (n < 0 || m < 1) return -1;
  int P = 0;
  for (int i = 0; i < n; ++i) {
    const double *yi = Y + (long)i * m;
    int keep = 1;
    for (int t = 0; t < m; ++t)
      if (!(yi[t] < ref[t])) keep = 0;
    for (int j = 0; j < n && keep; ++j) {
      if (j == i) continue;
      const double *yj = Y + (long)j * m;
      int all_le = 1, any_lt = 0, all_eq = 1;
      for (int t = 0; t < m; ++t) {
        if (yj[t] > yi[t]) all_le = 0;
        if (yj[t] < yi[t]) any_lt = 1;
        if (yj[t] != yi[t]) all_eq = 0;
      }
      if (all_le && any_lt) keep = 0;      /* j dominates i */
      if (all_eq && j < i) keep = 0;       /* duplicate: lowest index survives */
    }
    mask[i] = (unsigned char)keep;
    if (keep) order[P++] = i;
  }
  g_sortY = Y;
  g_sortM = m;
  qsort(order, (size_t)P, sizeof(int), cmp_lex);
  return P;
}

/* ---- Hypervolume by slicing ---------------------------------------------- */
long long bo_hv_scratch_size(int P, int m) {
  /* each recursion level copies at most P points of its dimension */
  return (long long)(P + 1) * m * (m + 1) + 16;
}

static int cmp_dbl2(const void *pa, const void *pb) { /* (f1, f2) lexicographic */
  const double *a = (const double *)pa, *b = (const double *)pb;
  if (a[0] != b[0]) return a[0] < b[0] ? -1 : 1;
  if (a[1] != b[1]) return a[1] < b[1] ? -1 : 1;
  return 0;
}

static _Thread_local int g_lastdim;
static int cmp_last(const void *pa, const void *pb) {
  const double *a = (const double *)pa, *b = (const double *)pb;
  double x = a[g_lastdim], y = b[g_lastdim];
  return (x > y) - (x < y);
}

/* pts: Q x m points, all strictly better than ref; may be reordered. */
static double hv_rec(double *pts, int Q, int m, const double *ref, double *scratch) {
  if (Q == 0) return 0.0;
  if (m == 1) {
    double lo = ref[0];
    for (int i = 0; i < Q; ++i)
      if (pts[i] < lo) lo = pts[i];
    return ref[0] - lo;
  }
  if (m == 2) { /* staircase sweep along f1 */
    qsort(pts, (size_t)Q, 2 * sizeof(double), cmp_dbl2);
    double hv = 0.0, cur = ref[1];
    for (int i = 0; i < Q; ++i) {
      if (pts[2 * i + 1] < cur) {
        hv += (ref[0] - pts[2 * i]) * (cur - pts[2 * i + 1]);
        cur = pts[2 * i + 1];
      }
    }
    return hv;
  }
  /* slice along the last objective: between consecutive levels the
   * cross-section is the (m-1)-D hypervolume of the points below the level */
  g_lastdim = m - 1;
  qsort(pts, (size_t)Q, (size_t)m * sizeof(double), cmp_last);
  double *sub = scratch, *rest = scratch + (long)Q * (m - 1);
  double hv = 0.0;
  for (int j = 0; j < Q; ++j) {
    double z0 = pts[(long)j * m + m - 1];
    double z1 = j + 1 < Q ? pts[(long)(j + 1) * m + m - 1] : ref[m - 1];
    if (z1 <= z0) continue;
    for (int i = 0; i <= j; ++i)
      memcpy(sub + (long)i * (m - 1), pts + (long)i * m, sizeof(double) * (m - 1));
    double a = hv_rec(sub, j + 1, m - 1, ref, rest);
    g_lastdim = m - 1; /* restore after recursion (the comparator is not reentrant) */
    hv += (z1 - z0) * a;
  }
  return hv;
}

double bo_hv(const double *F, int P, int m, const double *ref, double *scratch) {
  double *own = NULL;
  if (!scratch) {
    own = (double *)malloc(sizeof(double) * (size_t)bo_hv_scratch_size(P, m));
    scratch = own;
  }
  double *pts = scratch;
  int Q = 0;
  for (int i = 0; i < P; ++i) {
    int in = 1;
    for (int t = 0; t < m; ++t)
      if (!(F[(long)i * m + t] < ref[t])) in = 0;
    if (in) memcpy(pts + (long)(Q++) * m, F + (long)i * m, sizeof(double) * m);
  }
  double hv = hv_rec(pts, Q, m, ref, pts + (long)(P + 1) * m);
  free(own);
  return hv;
}

double bo_hvi(const double *F, int P, int m, const double *ref, const double *y) {
  double *all = (double *)malloc(sizeof(double) * (size_t)(P + 1) * m);
  memcpy(all, F, sizeof(double) * (size_t)P * m);
  memcpy(all + (long)P * m, y, sizeof(double) * m);
  double v = bo_hv(all, P + 1, m, ref, NULL) - bo_hv(F, P, m, ref, NULL);
  free(all);
  return v;
}

/* ---- closed-form 2-D EHVI ------------------------------------------------ */
static double std_cdf(double z) { return 0.5 * erfc(-z / sqrt(2.0)); }
static double std_pdf(double z) { return exp(-0.5 * z * z) / sqrt(2.0 * 3.14159265358979323846); }

/* psi(c) = E[(c - Y)_+], Y ~ N(mu, sigma^2); psi(-inf) = 0 */
static double psi(double c, double mu, double sigma) {
  if (isinf(c) && c < 0) return 0.0;
  if (!(sigma > 0.0)) return c > mu ? c - mu : 0.0;
  double z = (c - mu) / sigma;
  return (c - mu) * std_cdf(z) + sigma * std_pdf(z);
}

/* Constrained (Sec. 5.2 "Constrained qNEHVI", feasibility g_t = Y_t - c_t <= 0
 * on the minimised objectives): psi_c(v) = E[(v - Y)_+ 1[Y <= c]]. Since
 * (v - Y)_+ 1[Y <= c] = (v - Y) 1[Y <= w] with w = min(v, c),
 * psi_c(v) = (v - mu) Phi(z) + sigma phi(z), z = (w - mu) / sigma;
 * c = +infinity gives psi(v). */
static double psi_c(double v, double cons, double mu, double sigma) {
  if (isinf(v) && v < 0) return 0.0;
  double w = v < cons ? v : cons;
  if (!(sigma > 0.0)) return mu <= w ? v - mu : 0.0;
  double z = (w - mu) / sigma;
  return (v - mu) * std_cdf(z) + sigma * std_pdf(z);
}

void bo_ehvi2d(const double *mean, const double *var, long long N, const double *F,
               int P, const double *ref, const double *cons, double *acq, int nthreads) {
  int nt = nthreads_or_default(nthreads);
  const double c1 = cons ? cons[0] : INFINITY, c2 = cons ? cons[1] : INFINITY;
#pragma omp parallel for schedule(static) num_threads(nt)
  for (long long c = 0; c < N; ++c) {
    double mu1 = mean[2 * c], mu2 = mean[2 * c + 1];
    double sg1 = sqrt(var[2 * c]), sg2 = sqrt(var[2 * c + 1]);
    double e = 0.0;
    for (int i = 0; i <= P; ++i) {
      /* cell i: f1 in [a_i, b_i), f2 below u_i; with independent objectives
       * E[HVI 1[Y <= c]] factors per cell into the two objectives' terms */
      double a = i == 0 ? -INFINITY : F[2 * (i - 1)];
      double b = i == P ? ref[0] : F[2 * i];
      double u = i == 0 ? ref[1] : F[2 * (i - 1) + 1];
      if (cons)
        e += (psi_c(b, c1, mu1, sg1) - psi_c(a, c1, mu1, sg1)) * psi_c(u, c2, mu2, sg2);
      else
        e += (psi(b, mu1, sg1) - psi(a, mu1, sg1)) * psi(u, mu2, sg2);
    }
    acq[c] = e;
  }
}

/* ---- Monte-Carlo HVI ------------------------------------------------------ */
void bo_mc_hvi(const double *mean, const double *var, long long N, int m,
               const float *eps, int S, long long eps_stride, const double *F,
               int P, const double *ref, const double *cons, double *acq, int nthreads) {
  int nt = nthreads_or_default(nthreads);
  double hvF = bo_hv(F, P, m, ref, NULL);
  long long scr = bo_hv_scratch_size(P + 1, m);
#pragma omp parallel num_threads(nt)
  {
    double *all = (double *)malloc(sizeof(double) * (size_t)((P + 1) * m + m + scr));
    double *sg = all + (long)(P + 1) * m, *scratch = sg + m;
    memcpy(all, F, sizeof(double) * (size_t)P * m);
#pragma omp for schedule(dynamic, 64)
    for (long long c = 0; c < N; ++c) {
      for (int t = 0; t < m; ++t) sg[t] = sqrt(var[c * m + t]);
      double sum = 0.0;
      for (int s = 0; s < S; ++s) {
        int feasible = 1;
        for (int t = 0; t < m; ++t) {
          all[(long)P * m + t] =
              mean[c * m + t] + sg[t] * (double)eps[c * eps_stride + (long long)t * S + s];
          if (cons && !(all[(long)P * m + t] <= cons[t])) feasible = 0;
        }
        if (feasible) sum += bo_hv(all, P + 1, m, ref, scratch) - hvF;  /* else HVI x 0 */
      }
      acq[c] = sum / S;
    }
    free(all);
  }
}

/* ---- noisy expected hypervolume improvement (in-sample joint draws) --------- */
/* Lower Cholesky factor of the n x n matrix A in place (Cholesky-Banachiewicz);
 * the upper triangle is set to 0. Returns 2 when a pivot is not positive. */
static int chol_in_place(double *A, int n) {
  for (int i = 0; i < n; ++i) {
    for (int j = 0; j <= i; ++j) {
      double s = A[(long)i * n + j];
      for (int k = 0; k < j; ++k) s -= A[(long)i * n + k] * A[(long)j * n + k];
      if (i == j) {
        if (!(s > 0.0)) return 2;
        A[(long)i * n + i] = sqrt(s);
      } else {
        A[(long)i * n + j] = s / A[(long)j * n + j];
      }
    }
    for (int j = i + 1; j < n; ++j) A[(long)i * n + j] = 0.0;
  }
  return 0;
}

/* x = L^-1 b by forward substitution (L lower, n x n) */
static void fwd_subst(const double *L, int n, const double *b, double *x) {
  for (int i = 0; i < n; ++i) {
    double s = b[i];
    for (int k = 0; k < i; ++k) s -= L[(long)i * n + k] * x[k];
    x[i] = s / L[(long)i * n + i];
  }
}

int bo_joint_draws(const double *X, const double *y, int n, int d, const double *ls, double s2,
                   double noise, int dtau, const double *kc, double jitter, const float *z, int S,
                   const float *Xc, long long N, double *Yin, double *mean, double *cvar,
                   double *shift, int nthreads) {
  if (n < 1 || d < 1 || S < 1 || N < 0 || !X || !y || !ls || !z) return 1;
  const long nn = (long)n * n;
  double *L = (double *)malloc(sizeof(double) * nn), *alpha = (double *)malloc(sizeof(double) * n);
  double *Knn = (double *)malloc(sizeof(double) * nn), *V = (double *)malloc(sizeof(double) * nn);
  double *F = (double *)malloc(sizeof(double) * nn), *col = (double *)malloc(sizeof(double) * n);
  double *mu = (double *)malloc(sizeof(double) * n);
  int rc = bo_gp_fit_k(X, y, n, d, ls, s2, noise, dtau, kc, L, alpha);
  if (rc) goto done;
  /* the noise-free kernel matrix and V = L^-1 K_nn, column by column */
  for (int i = 0; i < n; ++i)
    for (int j = 0; j < n; ++j)
      Knn[(long)i * n + j] = bo_kernel(X + (long)i * d, X + (long)j * d, d, ls, s2, dtau, kc);
  for (int j = 0; j < n; ++j) {
    for (int i = 0; i < n; ++i) col[i] = Knn[(long)i * n + j];
    double *v = mu; /* scratch */
    fwd_subst(L, n, col, v);
    for (int i = 0; i < n; ++i) V[(long)i * n + j] = v[i];
  }
  /* in-sample posterior: mean K_nn alpha, covariance K_nn - K_nn K^-1 K_nn =
   * K_nn - V^T V, plus jitter * s2 on the diagonal; F its Cholesky factor */
  for (int i = 0; i < n; ++i) {
    double m_i = 0.0;
    for (int j = 0; j < n; ++j) m_i += Knn[(long)i * n + j] * alpha[j];
    mu[i] = m_i;
  }
  for (int i = 0; i < n; ++i)
    for (int j = 0; j < n; ++j) {
      double c = Knn[(long)i * n + j];
      for (int k = 0; k < n; ++k) c -= V[(long)k * n + i] * V[(long)k * n + j];
      F[(long)i * n + j] = c + (i == j ? jitter * s2 : 0.0);
    }
  rc = chol_in_place(F, n);
  if (rc) goto done;
  /* the in-sample draws mu + F z_s */
  for (int s = 0; s < S; ++s)
    for (int i = 0; i < n; ++i) {
      double v = mu[i];
      for (int j = 0; j <= i; ++j) v += F[(long)i * n + j] * (double)z[(long)s * n + j];
      Yin[(long)s * n + i] = v;
    }
  /* each candidate: marginal mean and variance, the cross-covariance with the
   * observed points Sigma_nx = k* - K_nn K^-1 k* = k* - V^T (L^-1 k*), its
   * coefficients l = F^-1 Sigma_nx on the in-sample normals, and the variance
   * left once the in-sample values are fixed, var - l^T l */
  {
    const int nt = nthreads_or_default(nthreads);
#pragma omp parallel num_threads(nt)
    {
      double *ks = (double *)malloc(sizeof(double) * (4 * (size_t)n + (size_t)d));
      double *v = ks + n, *sx = v + n, *l = sx + n, *xd = l + n;
#pragma omp for schedule(dynamic, 16)
      for (long long c = 0; c < N; ++c) {
        for (int k = 0; k < d; ++k) xd[k] = (double)Xc[c * d + k];
        for (int j = 0; j < n; ++j) ks[j] = bo_kernel(X + (long)j * d, xd, d, ls, s2, dtau, kc);
        const double kxx = bo_kernel(xd, xd, d, ls, s2, dtau, kc);
        double mc = 0.0;
        for (int j = 0; j < n; ++j) mc += ks[j] * alpha[j];
        fwd_subst(L, n, ks, v);
        double vv = 0.0;
        for (int j = 0; j < n; ++j) vv += v[j] * v[j];
        for (int i = 0; i < n; ++i) {
          double t = ks[i];
          for (int k = 0; k < n; ++k) t -= V[(long)k * n + i] * v[k];
          sx[i] = t;
        }
        fwd_subst(F, n, sx, l);
        double ll = 0.0;
        for (int j = 0; j < n; ++j) ll += l[j] * l[j];
        mean[c] = mc;
        cvar[c] = kxx - vv - ll;
        for (int s = 0; s < S; ++s) {
          double t = 0.0;
          for (int j = 0; j < n; ++j) t += l[j] * (double)z[(long)s * n + j];
          shift[c * S + s] = t;
        }
      }
      free(ks);
    }
  }
done:
  free(L); free(alpha); free(Knn); free(V); free(F); free(col); free(mu);
  return rc;
}

void bo_nehvi_mc(const double *Yin, int n, int m, int S, const double *mean, const double *cvar,
                 const double *shift, const float *eps, long long eps_stride, long long N,
                 const double *ref, const double *cons, double *acq, int nthreads) {
  /* per sample: the Pareto front of the feasible in-sample draws */
  double *fr = (double *)malloc(sizeof(double) * (size_t)S * n * m + 1);
  int *P = (int *)malloc(sizeof(int) * (size_t)S);
  double *hvF = (double *)malloc(sizeof(double) * (size_t)S);
  double *pts = (double *)malloc(sizeof(double) * (size_t)n * m + 1);
  unsigned char *mask = (unsigned char *)malloc((size_t)n + 1);
  int *order = (int *)malloc(sizeof(int) * (size_t)n + 1);
  for (int s = 0; s < S; ++s) {
    int q = 0;
    for (int i = 0; i < n; ++i) {
      const double *yi = Yin + ((long)s * n + i) * m;
      int ok = 1;
      for (int t = 0; t < m && cons; ++t)
        if (!(yi[t] <= cons[t])) ok = 0;
      if (ok) memcpy(pts + (long)(q++) * m, yi, sizeof(double) * m);
    }
    const int np = bo_pareto_front(pts, q, m, ref, mask, order);
    for (int k = 0; k < np; ++k)
      memcpy(fr + ((long)s * n + k) * m, pts + (long)order[k] * m, sizeof(double) * m);
    P[s] = np;
    hvF[s] = bo_hv(fr + (long)s * n * m, np, m, ref, NULL);
  }
  free(pts); free(mask); free(order);
  const int nt = nthreads_or_default(nthreads);
  long long scr = bo_hv_scratch_size(n + 1, m);
#pragma omp parallel num_threads(nt)
  {
    double *all = (double *)malloc(sizeof(double) * (size_t)((n + 1) * m + m + scr));
    double *sg = all + (long)(n + 1) * m, *scratch = sg + m;
#pragma omp for schedule(dynamic, 64)
    for (long long c = 0; c < N; ++c) {
      for (int t = 0; t < m; ++t) sg[t] = sqrt(cvar[c * m + t] > 0.0 ? cvar[c * m + t] : 0.0);
      double sum = 0.0;
      for (int s = 0; s < S; ++s) {
        const int np = P[s];
        memcpy(all, fr + (long)s * n * m, sizeof(double) * (size_t)np * m);
        int feasible = 1;
        for (int t = 0; t < m; ++t) {
          const double v = mean[c * m + t] + shift[(c * m + t) * S + s] +
                           sg[t] * (double)eps[c * eps_stride + (long long)t * S + s];
          all[(long)np * m + t] = v;
          if (cons && !(v <= cons[t])) feasible = 0;
        }
        if (feasible) sum += bo_hv(all, np + 1, m, ref, scratch) - hvF[s]; /* else HVI x 0 */
      }
      acq[c] = sum / S;
    }
    free(all);
  }
  free(fr); free(P); free(hvF);
}

/* ---- top-k ----------------------------------------------------------------- */
static _Thread_local const double *g_topv;
static int cmp_top(const void *pa, const void *pb) {
  long long a = *(const long long *)pa, b = *(const long long *)pb;
  double va = g_topv[a], vb = g_topv[b];
  if (isnan(va)) va = -INFINITY;
  if (isnan(vb)) vb = -INFINITY;
  if (va != vb) return va > vb ? -1 : 1;
  return (a > b) - (a < b);
}

void bo_topk(const double *acq, long long N, int k, long long *idx, double *val) {
  long long *ord = (long long *)malloc(sizeof(long long) * (size_t)(N > 0 ? N : 1));
  for (long long i = 0; i < N; ++i) ord[i] = i;
  g_topv = acq;
  qsort(ord, (size_t)N, sizeof(long long), cmp_top);
  for (int i = 0; i < k && i < N; ++i) {
    idx[i] = ord[i];
    val[i] = acq[ord[i]];
  }
  free(ord);
}
