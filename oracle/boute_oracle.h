/*
 * CPU oracle for the MOBO candidate-scoring step of BOute (arXiv 2602.10729).
 *
 * TEST INFRASTRUCTURE ONLY. This is a plain, slow, obviously correct fp64
 * restatement of what the scoring step computes, written from the paper, used
 * to check the CUDA library. Only the test suite, the package smoke check and
 * the benchmark's CPU-baseline leg may load it; the product path never does.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * Conventions: all matrices are row-major, contiguous; doubles unless noted.
 * Every objective is minimised (Sec. 4.3, problem formulation).
 * Return codes: 0 ok, 1 invalid argument, 2 matrix not positive definite.
 */
#ifndef BOUTE_ORACLE_H
#define BOUTE_ORACLE_H

#ifdef __cplusplus
extern "C" {
#endif

/* Outcome standardisation (Sec. 6, "Standardize" outcome transform):
 * Ys[:,t] = (Y[:,t] - mean_t) / std_t, std with the n-1 denominator; a column
 * with n < 2 or std < 1e-8 is divided by 1. Y, Ys: n x m. */
int bo_standardize(const double *Y, int n, int m, double *Ys);

/* ARD Matern-5/2 kernel with outputscale (Sec. 6 (i): MaternKernel nu=2.5
 * wrapped in ScaleKernel): s2 (1 + sqrt5 r + 5 r^2/3) exp(-sqrt5 r),
 * r^2 = sum_t ((a_t - b_t) / ls_t)^2. */
double bo_matern52(const double *a, const double *b, int d, const double *ls, double s2);

/* ARD Matern-3/2 kernel with outputscale (Sec. 6 (ii): MaternKernel nu=1.5):
 * s2 (1 + sqrt3 r) exp(-sqrt3 r), r as for bo_matern52. */
double bo_matern32(const double *a, const double *b, int d, const double *ls, double s2);

/* Preference weight of a deployment (Sec. 5.2 S5): w(c) = exp(beta sum_k
 * pref_k c_k), with c the allocation counts a_{m,n} flattened (dc entries) and
 * pref the matching entries s_{m,n} of the preference matrix. */
double bo_pref_weight(const double *c, int dc, double beta, const double *pref);

/* The GP's kernel. kc = NULL: the ARD Matern-5/2 kernel above (s2). Otherwise
 * the composite kernel of Sec. 5.2 ("Additive kernels", S5) as Sec. 6
 * assembles it, the routing features tau = x[0, dtau), the deployment
 * features c = x[dtau, d):
 *   k = s2 k52(tau, tau*) + kc[0] w(c) w(c*) k32(c, c*) + kc[1] k52(tau, tau*) k32(c, c*)
 * with k52, k32 the unscaled ARD Matern kernels (lengthscales ls[0, dtau) and
 * ls[dtau, d)), kc[0] and kc[1] the outputscales of the preference-weighted
 * deployment kernel and of the interaction (phi), kc[2] = beta and
 * kc[3 .. 3 + d - dtau) = pref. */
double bo_kernel(const double *a, const double *b, int d, const double *ls, double s2,
                 int dtau, const double *kc);

/* Outcome transforms before Standardize (Sec. 5.2 S4; Sec. 6): per objective
 * t, codes[t] & 3 = 0 identity, 1 log (latency), 2 logit (quality); bit 4
 * negates (a maximised outcome becomes a minimised one). codes = NULL: all
 * identity. Y, Yt: n x m. Values outside a transform's domain give NaN. */
int bo_outcome_transform(const double *Y, int n, int m, const int *codes, double *Yt);

/* Exact GP fit with fixed hyperparameters (Sec. 5.2 step (i); Sec. 6
 * SingleTaskGP, zero prior mean on standardised outcomes):
 * K = s2 M52(X, X) + noise I, L = chol(K) (Cholesky-Banachiewicz, no jitter),
 * alpha = K^-1 y by forward then back substitution.
 * X: n x d; y: n; ls: d; L: n x n (upper triangle set to 0); alpha: n.
 * Returns 2 when a pivot is not positive. */
int bo_gp_fit(const double *X, const double *y, int n, int d, const double *ls,
              double s2, double noise, double *L, double *alpha);
/* The same with the kernel bo_kernel(., ., d, ls, s2, dtau, kc). */
int bo_gp_fit_k(const double *X, const double *y, int n, int d, const double *ls, double s2,
                double noise, int dtau, const double *kc, double *L, double *alpha);

/* Latent-function posterior at fp32 candidates (cast to double):
 * mean = k*^T alpha, var = max(0, s2 - v^T v) with v = L^-1 k* by forward
 * substitution. Xc: N x d float; mean, var: N. nthreads <= 0: library default. */
void bo_gp_posterior(const double *X, int n, int d, const double *ls, double s2,
                     const double *L, const double *alpha, const float *Xc,
                     long long N, double *mean, double *var, int nthreads);
/* The same with the kernel bo_kernel(., ., d, ls, s2, dtau, kc); the prior
 * variance is k(x, x), which depends on x through the preference weight. */
void bo_gp_posterior_k(const double *X, int n, int d, const double *ls, double s2, int dtau,
                       const double *kc, const double *L, const double *alpha, const float *Xc,
                       long long N, double *mean, double *var, int nthreads);

/* Log marginal likelihood log p(y | X, theta) of the zero-mean GP with the
 * Matern-5/2 kernel above (Sec. 6: the hyperparameters are learned by
 * maximising it), -1/2 y^T K^-1 y - 1/2 log det K - n/2 log 2 pi, K = s2
 * M52(X, X) + noise I; NaN when K is not positive definite. grad (d + 2, or
 * NULL): its gradient with respect to theta = (log l_1 .. log l_d, log s2,
 * log noise), 1/2 tr((alpha alpha^T - K^-1) dK/dtheta_q). */
double bo_gp_mll(const double *X, const double *y, int n, int d, const double *ls, double s2,
                 double noise, double *grad);

/* Bounds of the learned log-parameters and the Adam constants of bo_gp_learn. */
#define BO_LOG_LS_MIN (-6.907755278982137)    /* log 1e-3 */
#define BO_LOG_LS_MAX (6.907755278982137)     /* log 1e3 */
#define BO_LOG_S2_MIN (-6.907755278982137)    /* log 1e-3 */
#define BO_LOG_S2_MAX (6.907755278982137)     /* log 1e3 */
#define BO_LOG_NOISE_MIN (-9.210340371976182) /* log 1e-4 */
#define BO_LOG_NOISE_MAX (2.302585092994046)  /* log 10 */
#define BO_LOG_SC_MIN (-9.210340371976182)    /* log 1e-4: s2_c, s2_x */
#define BO_LOG_SC_MAX (6.907755278982137)     /* log 1e3 */
#define BO_BETA_MIN (-3.0)
#define BO_BETA_MAX (3.0)
#define BO_ADAM_B1 0.9
#define BO_ADAM_B2 0.999
#define BO_ADAM_EPS 1e-8

/* Hyperparameter learning (Sec. 6): from each of R starting points
 * theta0[r] (d + 2 log-parameters, clamped to the bounds above), `iters`
 * steps of Adam ascent on bo_gp_mll with step size lr (bias-corrected first
 * and second moments, BO_ADAM_*), each step followed by the clamp. Writes the
 * final theta (R x (d + 2)), its log marginal likelihood mll (R) and, when
 * grad is not NULL, the gradient there (R x (d + 2)). A restart whose K stops
 * being positive definite keeps its last theta (mll NaN). */
int bo_gp_learn(const double *X, const double *y, int n, int d, const double *theta0, int R,
                int iters, double lr, double *theta, double *mll, double *grad);

/* The same two for the composite kernel (bo_kernel with kc): theta = (log
 * l_1..log l_d, log s2, log noise, log s2_c, log s2_x, beta), d + 5 values;
 * kc = [s2_c, s2_x, beta, pref...]; the extra bounds BO_LOG_SC_*, BO_BETA_*;
 * pref (d - dtau preference entries) stays fixed. grad: d + 5 values. */
double bo_gp_mll_k(const double *X, const double *y, int n, int d, const double *ls, double s2,
                   double noise, int dtau, const double *kc, double *grad);
int bo_gp_learn_k(const double *X, const double *y, int n, int d, int dtau, const double *pref,
                  const double *theta0, int R, int iters, double lr, double *theta, double *mll,
                  double *grad);

/* Monte-Carlo base normals from a counter-based generator (the MC estimate of
 * Sec. 5.2 needs standard normals; these are drawn reproducibly from a seed):
 * Philox4x64-10 (Salmon et al., SC'11) maps a 4 x 64-bit counter and a
 * 2 x 64-bit key to 4 x 64-bit words; bo_base_normals fills eps (B x N x m x
 * S fp32, the layout of boute_acq_mc_hvi) block by block: samples 4j..4j+3 of
 * candidate c, objective t, problem b come from counter (j, c, b m + t, 0)
 * and key (seed, 0), each word w giving the uniform ((w >> 11) + 1/2) 2^-53,
 * each pair (u1, u2) the normals sqrt(-2 ln u1) (cos 2 pi u2, sin 2 pi u2),
 * computed in fp64 and rounded to fp32. */
void bo_philox4x64(const unsigned long long ctr[4], const unsigned long long key[2],
                   unsigned long long out[4]);
void bo_base_normals(unsigned long long seed, int B, long long N, int m, int S, float *eps);

/* Pareto front of observed outcomes (Sec. 5.2, Pareto-optimal set; all
 * objectives minimised): point i is kept iff no j dominates it (Y_j <= Y_i in
 * every objective, < in one), no exact duplicate j < i exists, and
 * Y_i,t < ref_t for every t. mask: n bytes (1 = kept). order: the kept indices
 * sorted by f1, then f2, ..., then index. Returns P = number kept. */
int bo_pareto_front(const double *Y, int n, int m, const double *ref,
                    unsigned char *mask, int *order);

/* Hypervolume dominated by the points F (P x m) and bounded by ref, by
 * recursive slicing along the last objective with a 2-D staircase sweep at
 * the bottom. Points not strictly better than ref in every objective add
 * nothing. scratch: at least bo_hv_scratch_size(P, m) doubles, or NULL. */
double bo_hv(const double *F, int P, int m, const double *ref, double *scratch);
long long bo_hv_scratch_size(int P, int m);

/* Hypervolume improvement of y over F: HV(F u {y}) - HV(F). */
double bo_hvi(const double *F, int P, int m, const double *ref, const double *y);

/* Closed-form expected hypervolume improvement for two independent Gaussian
 * objectives (the expectation of HVI in Sec. 5.2 "Constrained qNEHVI", taken
 * in closed form over the P+1 cells of the sorted 2-D front):
 * EHVI = sum_i [psi1(b_i) - psi1(a_i)] psi2(u_i),
 * psi(c) = E[(c - Y)_+] = (c - mu) Phi(z) + sigma phi(z), z = (c - mu)/sigma.
 * cons (2 thresholds on the minimised objectives, or NULL): the feasibility
 * indicator 1[Y_1 <= c_1, Y_2 <= c_2] inside the expectation, which turns psi
 * into psi_c(v) = E[(v - Y)_+ 1[Y <= c]].
 * mean, var: N x 2; F: P x 2 sorted by f1 ascending; acq: N. */
void bo_ehvi2d(const double *mean, const double *var, long long N, const double *F,
               int P, const double *ref, const double *cons, double *acq, int nthreads);

/* Monte-Carlo hypervolume improvement (Sec. 5.2: expectation of HVI over
 * posterior samples, by Monte-Carlo integration): sample s of candidate c is
 * y_t = mean_t + sqrt(var_t) eps[c*eps_stride + t*S + s]; acq = mean over the
 * S samples of HV(F u {y}) - HV(F), each multiplied by the feasibility
 * indicator 1[y_t <= cons_t for every t] when cons (m thresholds) is given.
 * mean, var: N x m; eps: float. */
void bo_mc_hvi(const double *mean, const double *var, long long N, int m,
               const float *eps, int S, long long eps_stride, const double *F,
               int P, const double *ref, const double *cons, double *acq, int nthreads);

/* Joint posterior draws for the noisy acquisition (Sec. 5.2, constrained
 * qNEHVI: the expectation runs over samples of the joint posterior, here of
 * the objective at the n observed points and at each candidate, so that the
 * front the candidate improves on is itself a posterior draw). One objective,
 * the fit of bo_gp_fit_k. For S in-sample normals z (S x n float):
 *   Yin[s] = mu_n + F z_s, mu_n = K_nn alpha, F = chol(K_nn - K_nn K^-1 K_nn
 *   + jitter s2 I) (K_nn the noise-free kernel matrix, K = K_nn + noise I);
 * and for each candidate x (Xc: N x d float) the marginal mean, the
 * cross-covariance Sigma_nx = k* - K_nn K^-1 k*, l = F^-1 Sigma_nx, and
 *   cvar = k(x, x) - k*^T K^-1 k* - l^T l,  shift[x][s] = l^T z_s,
 * so that the joint draw at x is mean + shift_s + sqrt(cvar) eps_s: the
 * Cholesky factor of the joint covariance of (f(X), f(x)) with the jitter on
 * the in-sample block, applied to (z_s, eps_s). Yin: S x n; mean, cvar: N;
 * shift: N x S. Returns 2 when K or the in-sample covariance is not positive
 * definite. nthreads <= 0: library default. */
int bo_joint_draws(const double *X, const double *y, int n, int d, const double *ls, double s2,
                   double noise, int dtau, const double *kc, double jitter, const float *z, int S,
                   const float *Xc, long long N, double *Yin, double *mean, double *cvar,
                   double *shift, int nthreads);

/* Monte-Carlo noisy expected hypervolume improvement (Sec. 5.2, constrained
 * qNEHVI with q = 1): for each sample s the front is the Pareto front
 * (bo_pareto_front against ref) of the in-sample draws Yin[s] (n x m) that
 * satisfy the constraints (y_t <= cons[t] for every t; all of them when cons
 * is NULL); the candidate's draw y_t = mean_t + shift_t,s + sqrt(max(cvar_t,
 * 0)) eps_t,s counts its hypervolume improvement over that front when it is
 * feasible itself; acq = the average over the S samples. Yin: S x n x m;
 * mean, cvar: N x m; shift: N x m x S; eps: float, candidate c's block at
 * c * eps_stride, (m, S) row-major. */
void bo_nehvi_mc(const double *Yin, int n, int m, int S, const double *mean, const double *cvar,
                 const double *shift, const float *eps, long long eps_stride, long long N,
                 const double *ref, const double *cons, double *acq, int nthreads);

/* Top-k selection (Sec. 5.2 step (ii): the next configuration is the best
 * scored candidate): the first k entries of the order (value descending, NaN
 * as -infinity, equal values by ascending index). idx, val: k. */
void bo_topk(const double *acq, long long N, int k, long long *idx, double *val);

/* Number of OpenMP threads a call with nthreads <= 0 uses. */
int bo_default_threads(void);

#ifdef __cplusplus
}
#endif
#endif
