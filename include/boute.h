/*
 * libboute: GB300-native candidate scoring for the multi-objective Bayesian
 * optimisation (MOBO) loop of BOute (arXiv 2602.10729).
 *
 * One MOBO iteration (Sec. 5.2, "Overall MOBO workflow") fits one Gaussian
 * process per objective, then optimises the hypervolume-improvement
 * acquisition (Sec. 5.2, "Constrained qNEHVI") over the decision space and
 * selects the next configuration theta*. This library implements that step
 * over a discrete candidate set: standardise -> fit -> Pareto front ->
 * posterior -> acquisition -> top-k. All objectives are minimised (Sec. 4.3).
 *
 * Conventions (every entry point):
 *  - Arrays are DEVICE pointers, owned by the caller, row-major and
 *    contiguous, unless the argument says "host". Only boute_gp and
 *    boute_engine objects own device memory, freed by their *_free call.
 *  - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream) unless it says it synchronises.
 *  - Argument errors are returned synchronously and launch nothing. Errors
 *    raised on the device (a non-positive Cholesky pivot, a wait that timed
 *    out) are recorded in a device status word and returned by the next call
 *    that synchronises (boute_gp_status, boute_engine_step*).
 *  - B independent problems share one call; problem b's data follow
 *    problem b-1's in every array.
 *  - Limits: d <= 32, m <= 4 (m <= 3 for Monte-Carlo HVI, m == 2 for the
 *    closed-form EHVI), 1 <= n <= 2048, B*N < 2^31, k <= 1024.
 *
 * Status codes are the boute_status values; every function returns one.
 */
#ifndef BOUTE_H
#define BOUTE_H

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  BOUTE_OK = 0,
  BOUTE_ERR_INVALID_ARG = 1, /* bad size, null pointer, unsupported shape */
  BOUTE_ERR_NOT_PD = 2,      /* kernel matrix not positive definite */
  BOUTE_ERR_CUDA = 3,        /* a CUDA runtime call failed */
  BOUTE_ERR_OOM = 4,         /* device allocation failed */
  BOUTE_ERR_UNSUPPORTED = 5, /* no sm_103a device, or shape beyond the limits */
  BOUTE_ERR_TIMEOUT = 6      /* a device-side wait gave up (nothing hung) */
} boute_status;

typedef enum { BOUTE_ACQ_EHVI2D = 0, BOUTE_ACQ_MC_HVI = 1, BOUTE_ACQ_NEHVI = 2 } boute_acq_mode;

/* Human-readable name of a status code (static string). */
const char *boute_status_string(int status);

/* Number of kernels this library has launched in this process (all streams).
 * A monotone counter; differences bracket a region of work. */
unsigned long long boute_launch_count(void);

/* ---- outcome transforms and standardisation ------------------------------
 * Sec. 5.2 S4 and Sec. 6 (outcome transforms Log / Logit, then "Standardize"):
 * each raw outcome is first transformed per objective, transforms[t] & 3 =
 * BOUTE_TF_IDENTITY (0), BOUTE_TF_LOG (1, latency) or BOUTE_TF_LOGIT (2,
 * quality, log(y / (1 - y))), | BOUTE_TF_NEGATE (4) to minimise a maximised
 * outcome; then Ys[b,:,t] = (z[b,:,t] - mean) / std, std with the n-1
 * denominator; a column with n < 2 or std < 1e-8 is divided by 1.
 * transforms: HOST array of m codes, or NULL (all identity); an unknown code
 * is INVALID_ARG; outcomes outside a transform's domain give NaN.
 * Y, Ys: B x n x m fp64 (may alias). m <= 4. */
#define BOUTE_TF_IDENTITY 0
#define BOUTE_TF_LOG 1
#define BOUTE_TF_LOGIT 2
#define BOUTE_TF_NEGATE 4
int boute_standardize(const double *Y, int B, int n, int m, const int *transforms, double *Ys,
                      void *stream);

/* ---- GP fit ----------------------------------------------------------------
 * Sec. 5.2 step (i) and Sec. 6: one exact GP per objective (SingleTaskGP
 * models combined as a ModelListGP), ARD Matern-5/2 covariance with an
 * outputscale (MaternKernel nu=2.5 in a ScaleKernel), zero prior mean on
 * standardised outcomes, fixed hyperparameters:
 *   K = s2 * M52(X, X) + noise * I,  L = chol(K) (fp64, no jitter),
 *   the library keeps L^-1 and alpha = K^-1 y as the tensor-core operand of
 *   the posterior contraction.
 * boute_gp_create allocates a handle for B problems x m objectives of n
 * points in d dimensions (the only allocating call of the fit path);
 * boute_gp_fit recomputes it asynchronously from
 *   X: B x n x d fp64; Ys: B x n x m fp64 (standardised outcomes);
 *   lengthscale: B x m x d fp64; outputscale, noise: B x m fp64.
 * boute_gp_status synchronises `stream` and returns BOUTE_ERR_NOT_PD if a
 * pivot of any problem/objective was not positive (its posterior is then
 * undefined), else the first recorded device error, else BOUTE_OK; it clears
 * the recorded status. */
typedef struct boute_gp boute_gp;
int boute_gp_create(int B, int n, int d, int m, boute_gp **out);
int boute_gp_fit(boute_gp *gp, const double *X, const double *Ys, const double *lengthscale,
                 const double *outputscale, const double *noise, void *stream);
int boute_gp_status(boute_gp *gp, void *stream);
void boute_gp_free(boute_gp *gp);
/* ---- precision tiers ----------------------------------------------------------
 * Sec. 6 and Appendix C: the paper's MOBO runs its GP kernels in double
 * precision. BOUTE_PREC_FP32 (the default) is the fp32-accurate path of
 * boute_gp_posterior (posterior mean and variance within 1e-5 of the fp64
 * values). boute_gp_set_precision(gp, BOUTE_PREC_FP64) makes the handle's
 * later fits also compute K, its Cholesky factor L, W = L^-1 and alpha in
 * fp64 (on the CUDA cores; GB300's fp64 rate is a small fraction of its fp32
 * rate, so this tier serves accuracy, not throughput), and
 * boute_gp_posterior_fp64 then writes
 *   mean = k*^T alpha,  var = max(0, s2 - ||W k*||^2)
 * in fp64: Xc as for boute_gp_posterior; mean, var: B x m x N fp64 device
 * arrays. The FP64 tier serves n <= 128 and the Matern-5/2 kernel: other
 * handles return BOUTE_ERR_UNSUPPORTED from set_precision (and set_kernel
 * with the composite kernel returns it for an FP64 handle); allocates its
 * fp64 buffers on the first switch. boute_gp_posterior_fp64 on a handle not
 * set to FP64 is INVALID_ARG; the fp32 path keeps working on an FP64 handle. */
#define BOUTE_PREC_FP32 0
#define BOUTE_PREC_FP64 1
int boute_gp_set_precision(boute_gp *gp, int prec);
int boute_gp_posterior_fp64(const boute_gp *gp, const float *Xc, long long N, double *mean,
                            double *var, void *stream);
/* The paper's composite kernel for the handle's later fits and posteriors
 * (Sec. 5.2 "Additive kernels" with the preference weighting of S5, as
 * Sec. 6 assembles it: k_tau + k~_c + k_x, each in its own ScaleKernel):
 * the first d_tau features are routing features tau, the other d - d_tau
 * deployment features c (GPU counts a_{m,n}, flattened), and
 *   k(x, x*) = s2 k52(tau, tau*) + s2_c w(c) w(c*) k32(c, c*)
 *              + s2_x k52(tau, tau*) k32(c, c*),
 *   w(c) = exp(beta sum_k s_k c_k),
 * k52 / k32 the unscaled ARD Matern-5/2 / 3/2 kernels with the fit's
 * lengthscales of the respective features, s2 the fit's outputscale.
 * params: HOST array B x m x (3 + d - d_tau) fp64, per problem-objective
 * [s2_c, s2_x (the interaction weight phi), beta, s_0 .. s_{d-d_tau-1}]
 * (the preference-matrix entries matching the deployment features); copied
 * into the handle. params = NULL restores the Matern-5/2 kernel. The prior
 * variance k(x, x) = s2 + s2_x + s2_c w(c)^2 depends on the candidate.
 * Waits for all work on the device first. */
int boute_gp_set_kernel(boute_gp *gp, int d_tau, const double *params);

/* ---- hyperparameters ----------------------------------------------------------
 * Sec. 6: the lengthscales, outputscale and noise are learned by maximising
 * the GP's log marginal likelihood (in double precision):
 *   log p(y | theta) = -1/2 y^T K^-1 y - 1/2 log det K - n/2 log 2 pi,
 *   K = s2 M52(X, X) + noise I,
 * over theta = (log l_1 .. log l_d, log s2, log noise). For every problem b,
 * objective t and restart r, `iters` steps of Adam ascent (bias-corrected
 * moments, BOUTE_ADAM_B1 / B2 / EPS, step size lr) from theta0, each step
 * followed by a clamp to the BOUTE_LOG_* bounds; then the log likelihood at
 * the final theta. The gradient is
 *   1/2 sum_ij (alpha_i alpha_j - K^-1_ij) dK_ij / dtheta_q,  alpha = K^-1 y.
 *   X: B x n x d fp64; Ys: B x n x m fp64 (standardised outcomes);
 *   theta0: B x m x R x (d + 2) fp64 starting points; theta (out, same
 *   layout): the final log-parameters; mll (out): B x m x R; grad (out,
 *   optional, same layout as theta): the gradient at the final theta.
 *   All device pointers; iters >= 0 (0: evaluate at theta0); R >= 1.
 * A restart whose K is not positive definite stops there: its theta is kept
 * and its mll (and grad) are NaN. One block per (b, t, r); a block's n x n
 * workspace is in shared memory up to n = 150 or so, else in stream-ordered
 * pool memory. Asynchronous on `stream`. */
#define BOUTE_LOG_LS_MIN (-6.907755278982137)    /* log 1e-3 */
#define BOUTE_LOG_LS_MAX (6.907755278982137)     /* log 1e3 */
#define BOUTE_LOG_S2_MIN (-6.907755278982137)    /* log 1e-3 */
#define BOUTE_LOG_S2_MAX (6.907755278982137)     /* log 1e3 */
#define BOUTE_LOG_NOISE_MIN (-9.210340371976182) /* log 1e-4 */
#define BOUTE_LOG_NOISE_MAX (2.302585092994046)  /* log 10 */
#define BOUTE_LOG_SC_MIN (-9.210340371976182)    /* log 1e-4: s2_c, s2_x */
#define BOUTE_LOG_SC_MAX (6.907755278982137)     /* log 1e3 */
#define BOUTE_BETA_MIN (-3.0)
#define BOUTE_BETA_MAX (3.0)
#define BOUTE_ADAM_B1 0.9
#define BOUTE_ADAM_B2 0.999
#define BOUTE_ADAM_EPS 1e-8
int boute_gp_learn(const double *X, const double *Ys, int B, int n, int d, int m,
                   const double *theta0, int R, int iters, double lr, double *theta,
                   double *mll, double *grad, void *stream);
/* The same for the composite kernel (boute_gp_set_kernel): theta = (log l_1
 * .. log l_d, log s2, log noise, log s2_c, log s2_x, beta), d + 5 values per
 * (b, t, r), the extra ones clamped to BOUTE_LOG_SC_* and BOUTE_BETA_*;
 * pref: B x m x (d - d_tau) fp64 device preference entries (held fixed). The
 * gradient adds
 *   dK/dlog l_q = (5/3)(1 + sqrt5 r_t) e^(-sqrt5 r_t) z_q^2 (s2 + s2_x k32)  (routing)
 *               = 3 e^(-sqrt3 r_c) z_q^2 (s2_c w_i w_j + s2_x k52)        (deployment),
 *   dK/dlog s2_c = s2_c w_i w_j k32, dK/dlog s2_x = s2_x k52 k32,
 *   dK/dbeta = s2_c w_i w_j k32 (<s, c_i> + <s, c_j>). */
int boute_gp_learn_k(const double *X, const double *Ys, int B, int n, int d, int m, int d_tau,
                     const double *pref, const double *theta0, int R, int iters, double lr,
                     double *theta, double *mll, double *grad, void *stream);

/* ---- posterior ---------------------------------------------------------------
 * Latent-function posterior of every objective at N candidates per problem
 * (Sec. 5.2: the acquisition is taken over the GP posterior):
 *   mean = K* alpha,  var = max(0, s2 - rowsum((K* L^-T)^2)),
 * with the Matern-5/2 cross-covariance K* built tile by tile in shared memory
 * and contracted on the tensor cores as fp16 hi/lo parts (three products per
 * term, fp32 accumulate: fp32-accurate) without ever being written to HBM.
 * The mean is reduced from the fp32 K* with compensated sums; a candidate
 * whose terms K*_j alpha_j add up to more than 256 times the mean's scale
 * (an ill-conditioned K) has its mean recomputed in fp64.
 *   Xc: B x N x d fp32 candidates (points of [0,1]^d or any real values);
 *   mean, var: B x m x N fp32 (objective-major per problem). */
int boute_gp_posterior(const boute_gp *gp, const float *Xc, long long N, float *mean,
                       float *var, void *stream);

/* ---- Pareto front and box decomposition -------------------------------------
 * Sec. 5.2 (Pareto-optimal set; Sec. 4.3, minimisation): point i of problem b
 * is on the front iff no point dominates it (<= in every objective, < in
 * one), no exact duplicate with a smaller index exists, and it is strictly
 * better than ref in every objective.
 *   Ys: B x n x m fp64; ref: B x m fp64;
 *   mask: B x n bytes (1 = on the front);
 *   front: B x n x m fp64, rows [0, P[b]) = the front sorted by f1, then f2,
 *          ..., then index (rows beyond P[b] are left unspecified);
 *   P: B ints. */
int boute_pareto_front(const double *Ys, int B, int n, int m, const double *ref,
                       unsigned char *mask, double *front, int *P, void *stream);

/* Disjoint boxes covering the region that improves on the front and is below
 * ref ({z <= ref : no front point p <= z}), the region whose volume inside
 * [y, ref] is the hypervolume improvement of y (Sec. 5.2). m = 2: the P+1
 * strips of the staircase; m = 3: a sweep along f3 (at most 2P+1 boxes).
 * Lower bounds may be -infinity.
 *   front, P: as written by boute_pareto_front (capacity n rows per problem);
 *   lower, upper: B x (2n+2) x m fp32; K: B ints (boxes per problem). */
int boute_box_decompose(const double *front, const int *P, int B, int n, int m,
                        const double *ref, float *lower, float *upper, int *K, void *stream);

/* ---- acquisition --------------------------------------------------------------
 * Expected hypervolume improvement (Sec. 5.2, "Constrained qNEHVI": the
 * expectation of HVI over the posterior), for m = 2 independent objectives in
 * closed form over the P+1 staircase cells:
 *   EHVI = sum_i [psi1(b_i) - psi1(a_i)] psi2(u_i),  psi(c) = E[(c - Y)_+].
 *   mean, var: B x 2 x N fp32 (boute_gp_posterior's layout);
 *   front, P: boute_pareto_front's output, n = its row capacity; ref: B x 2;
 *   cons: NULL, or B x 2 fp64 device thresholds k_t on the minimised
 *         (standardised) objectives, in the units of ref: the constrained
 *         acquisition of Sec. 5.2, E[HVI(Y) 1[Y_1 <= k_1] 1[Y_2 <= k_2]], which
 *         replaces psi_t by psi_t^c(c) = E[(c - Y_t)_+ 1[Y_t <= k_t]]; an
 *         infinite threshold constrains nothing; NaN is not a threshold (not
 *         checked on the device);
 *   acq: B x N fp32. */
int boute_acq_ehvi(const float *mean, const float *var, int B, long long N, const double *front,
                   const int *P, int n, const double *ref, const double *cons, float *acq,
                   void *stream);

/* Monte-Carlo hypervolume improvement (Sec. 5.2: the expectation estimated by Monte-Carlo
 * integration over posterior samples): sample s of candidate c is
 * y_t = mean_t + sqrt(var_t) * eps[c][t][s]; acq = mean over S samples of the
 * exact HVI of y, the volume of [y, ref] inside the boxes.
 *   lower, upper, K, box_cap: boute_box_decompose's output (box_cap = 2n+2);
 *   eps: fp32 base normals, candidate c of problem b at
 *        eps + (b*N + c) * eps_cand_stride, laid out m x S; eps_cand_stride =
 *        m*S for per-candidate normals, 0 for normals shared by all candidates
 *        of a problem (then problem b's block is at eps + b*m*S);
 *   cons: NULL, or B x m fp64 device thresholds (as for boute_acq_ehvi): a
 *         sample with some y_t > k_t contributes zero (HVI times the
 *         feasibility indicator, the constrained estimate of Sec. 5.2); the
 *         comparison is made in fp32;
 *   acq: B x N fp32. 2 <= m <= 3, 1 <= S. */
int boute_acq_mc_hvi(const float *mean, const float *var, int B, long long N, int m,
                     const float *lower, const float *upper, const int *K, int box_cap,
                     const float *eps, int S, long long eps_cand_stride, const double *cons,
                     float *acq, void *stream);

/* ---- noisy acquisition: in-sample joint draws ------------------------------------
 * Sec. 5.2, "Constrained qNEHVI" (q = 1): the expectation runs over samples of
 * the JOINT posterior of each objective at the n observed points X and at the
 * candidate, so that the front a candidate improves on is itself a posterior
 * draw (the observations are noisy). Draw s of objective t uses the Cholesky
 * factor of the joint covariance, with a jitter of 1e-8 * outputscale on the
 * in-sample block, applied to the normals (z_s, eps_s):
 *   Yin_s = mu_n + F z_s,  mu_n = K_nn alpha,
 *   F = chol(K_nn - K_nn K^-1 K_nn + 1e-8 s2 I)   (K = K_nn + noise I)
 *   y_s(x) = mean(x) + l(x)^T z_s + sqrt(cvar(x)) eps_s,  l = F^-1 Sigma_nx,
 *   cvar = k(x, x) - k*^T K^-1 k* - l^T l,  Sigma_nx = k* - K_nn K^-1 k*.
 * The per-candidate terms are contractions of k* (l^T z_s = k*^T G_s with
 * G = noise K^-1 F^-T Z), computed by the posterior's tensor-core kernel as
 * extra output columns.
 *
 * boute_gp_set_insample(gp, S): the handle's later fits prepare S in-sample
 * draws (1 <= S <= 1024; 0 turns them off). It re-plans the operand images,
 * which are then zero: fit again before the next insample or posterior call.
 * Allocates; waits for all work on the device. n (the handle's capacity)
 * <= 128 and the FP32 tier, else BOUTE_ERR_UNSUPPORTED.
 * boute_gp_insample, after boute_gp_fit with the same Ys, outputscale and
 * noise (B x n x m, B x m, B x m fp64): reads z (B x m x S x n fp32 standard
 * normals) and writes Yin (B x m x S x n fp32), and prepares the handle's
 * shift operands. A factor that is not positive definite records
 * BOUTE_ERR_NOT_PD (boute_gp_status).
 * boute_gp_posterior_joint: mean and cvar as boute_gp_posterior's mean and
 * var (B x m x N fp32; cvar clamped at 0) and shift[b][t][s][c] = l(x_c)^T z_s
 * (B x m x S x N fp32). boute_gp_posterior on such a handle still gives the
 * plain posterior. */
int boute_gp_set_insample(boute_gp *gp, int S);
int boute_gp_insample(boute_gp *gp, const double *Ys, const double *outputscale,
                      const double *noise, const float *z, float *Yin, void *stream);
int boute_gp_posterior_joint(const boute_gp *gp, const float *Xc, long long N, float *mean,
                             float *cvar, float *shift, void *stream);
/* The front of each in-sample draw (two objectives): the Pareto front,
 * against ref (B x 2 fp64), of the draw's points that meet the constraints
 * (cons: NULL or B x 2 fp64 thresholds, y_t <= cons_t) as the vertical strips
 * of the region it leaves undominated. Yin: B x 2 x S x n fp32 (n <= 128);
 * strips: B x S x (n + 1) x 4 fp32, strip j of draw s = (l1, u1, u2, 0): the
 * cells [l1, u1) x (-inf, u2), sorted by l1 (strip 0 has l1 = -inf);
 * counts: B x S int, the strips of each draw (front size + 1). */
int boute_insample_fronts(const float *Yin, int B, int n, int S, const double *ref,
                          const double *cons, float *strips, int *counts, void *stream);
/* Noisy MC hypervolume improvement (two objectives): draw s of candidate c
 * is y_t = mean_t + shift_t,s + sqrt(cvar_t) eps_t,s (eps laid out as for
 * boute_acq_mc_hvi); with cons, a draw counts only when y_t <= cons_t for
 * both t (fp32 comparison); its improvement is the area of [y, ref] inside
 * draw s's strips: sum_j (u1_j - max(l1_j, y_1))+ (u2_j - y_2)+; acq (B x N
 * fp32) = the mean over the S draws. mean, cvar, shift: the layouts of
 * boute_gp_posterior_joint; strips, counts, n: boute_insample_fronts's. */
int boute_acq_nehvi2d(const float *mean, const float *cvar, const float *shift, int B,
                      long long N, int S, const float *eps, long long eps_cand_stride,
                      const float *strips, const int *counts, int n, const double *cons,
                      float *acq, void *stream);

/* Optimising the acquisition over the decision space (Sec. 5.2 step (ii):
 * the acquisition is optimised to pick the next configuration; BoTorch does
 * it by gradient ascent from the best of many raw samples). Two objectives,
 * the Matern-5/2 kernel, the fitted handle `gp` (B problems); the
 * acquisition is the sample-average Monte-Carlo hypervolume improvement over
 * the observed front with base normals eps shared by every point,
 *   A(x) = (1/S) sum_s HVI(mean(x) + sd(x) eps_s),
 * differentiated through the posterior (k*, W = L^-1 and alpha of the fit).
 * From each starting point, `steps` steps of projected Adam ascent (beta1
 * 0.9, beta2 0.999, eps 1e-8, step size lr), every iterate clamped to
 * [xlo, xhi]; then the value and gradient at the final point.
 *   lower, upper, K, box_cap: boute_box_decompose's output for the front;
 *   eps: 2 x S fp32 (objective-major); X0: B x P x d fp32 starting points;
 *   xlo, xhi: d fp32 bounds; X: B x P x d fp32 final points; acq: B x P fp32
 *   their acquisition values; grad: B x P x d fp32 gradients there, or NULL.
 * steps = 0 evaluates the acquisition and its gradient at X0. Other kernels
 * or m != 2: BOUTE_ERR_UNSUPPORTED. */
int boute_acq_optimize(const boute_gp *gp, const float *lower, const float *upper, const int *K,
                       int box_cap, const float *eps, int S, const float *X0, int P,
                       const float *xlo, const float *xhi, int steps, float lr, float *X,
                       float *acq, float *grad, void *stream);

/* Failure detection: every device-side wait of the library is bounded (about
 * 2 s) and a wait that runs out records BOUTE_ERR_TIMEOUT in the call's
 * status instead of hanging. This self-test runs one such bounded wait on
 * an mbarrier with limit_ns (<= 2e9) and returns BOUTE_ERR_TIMEOUT when the
 * wait ran out (complete = 0: nothing arrives) or BOUTE_OK when it
 * completed (complete != 0: the one expected arrival is made). Synchronous;
 * the device stays usable either way. */
int boute_selftest_wait(int complete, unsigned long long limit_ns, void *stream);

/* Debug build (the library compiled with BOUTE_DEBUG_BOUNDS, see the
 * package's build_debug): the kernels check their index arithmetic — every
 * guarded access tests 0 <= index < extent, records the first index out of
 * its extent per source unit and skips the access (the bulk copies, the
 * operand images, the outputs, the strips and boxes, the selection). This
 * call waits for the device, returns 1 and fills rec (4 words: the source
 * unit 1 posterior, 2 in-sample, 3 acquisition, 4 front, 5 fit, 6 top-k;
 * the source line; the index; the extent) when some unit recorded one since
 * the last call, else 0; it clears the records. The product library returns
 * BOUTE_ERR_UNSUPPORTED (its checks compile to nothing). */
int boute_bounds_report(long long *rec);

/* Monte-Carlo base normals from a counter-based generator, for callers that
 * do not draw their own: Philox4x64-10 (Salmon et al., SC'11, counter-based:
 * any sample can be regenerated alone) and the Box-Muller transform in fp64,
 * rounded to fp32. eps: B x N x m x S device (the layout of
 * boute_acq_mc_hvi with eps_cand_stride = m*S); samples 4j..4j+3 of candidate
 * c, objective t, problem b come from counter (j, c, b m + t, 0) and key
 * (seed, 0), each 64-bit word w giving the uniform ((w >> 11) + 1/2) 2^-53
 * and each pair (u1, u2) the normals sqrt(-2 ln u1) (cos 2 pi u2, sin 2 pi u2).
 * Asynchronous on `stream`. */
int boute_base_normals(unsigned long long seed, int B, long long N, int m, int S, float *eps,
                       void *stream);

/* ---- selection ----------------------------------------------------------------
 * Sec. 5.2 step (ii): the next configuration(s) to evaluate are the best
 * scored candidates. Per problem, the k largest acq values in the order
 * (value descending, NaN as -infinity, -0 as +0, equal values by ascending
 * index); idx: B x k int64 (candidate index within its problem), val: B x k
 * fp32 (the acq value at idx). k <= min(N, 1024). Uses stream-ordered
 * scratch from the CUDA memory pool. */
int boute_select_topk(const float *acq, int B, long long N, int k, long long *idx, float *val,
                      void *stream);

/* boute_select_topk_noalloc: the same selection, bit for bit, with its
 * intermediate keys in a fixed array compiled into the library
 * (BOUTE_TOPK_NOALLOC_SCRATCH_BYTES of device memory, 8 MiB) instead of
 * memory from the CUDA pool; the paper has no counterpart, it is a service to
 * callers that must not allocate device memory on the call path: a caller
 * whose allocator already holds the device's free memory, a latency-critical
 * loop that cannot take the synchronisation cudaFree implies, or a fixed
 * memory budget. The call makes no allocation of any kind.
 *   Limit: 2 * B * ceil(N / 2048) * max(k, 32) * 8 bytes of scratch (0 when
 *   N <= 2048) must not exceed BOUTE_TOPK_NOALLOC_SCRATCH_BYTES; a larger
 *   request returns BOUTE_ERR_UNSUPPORTED before launching anything. Other
 *   argument errors are those of boute_select_topk.
 *   Set-up: the first call on a device, made with that device current, looks
 *   up the array's device address (once per device, under a lock); make that
 *   first call before any stream capture begins.
 *   The few words of the array that must start at zero (one counter per
 *   problem) are cleared by the call itself, on `stream`, before its kernel
 *   runs; every key is written before it is read.
 *   There is ONE array per device: calls that overlap in time on that device
 *   (on different streams, or from different threads) race on it and may
 *   return wrong results. Serialise them, e.g. by issuing them on one stream. */
#define BOUTE_TOPK_NOALLOC_SCRATCH_BYTES (8u << 20)
int boute_select_topk_noalloc(const float *acq, int B, long long N, int k, long long *idx,
                              float *val, void *stream);

/* ---- the whole scoring step ---------------------------------------------------
 * An engine owns every intermediate buffer of one workload shape and runs the
 * whole step: GP fit, then posterior, acquisition and selection on `stream`;
 * the front stage (standardise, Pareto front, boxes) on an internal second
 * stream forked from `stream` and joined back before the acquisition.
 * boute_engine_step: device inputs; boute_engine_step_host: HOST inputs and
 * outputs (copied in and out on `stream` inside the call); both synchronise
 * and return the fit status or the first device error.
 *   X: B x n x d fp64; Y: B x n x m fp64 raw outcomes (standardised inside);
 *   lengthscale: B x m x d; outputscale, noise: B x m; ref: B x m (fp64);
 *   Xc: B x N x d fp32; eps: B x N x m x S fp32 (modes MC_HVI and NEHVI; NULL
 *   otherwise);
 *   idx: B x k int64, val: B x k fp32.
 * boute_engine_step_async: as boute_engine_step without the final
 * synchronisation (device errors surface at the next synchronising call).
 * boute_engine_step_host_async: as boute_engine_step_host without the final
 * synchronisation, for a stream of steps: consecutive calls alternate between
 * two sets of device input buffers, so that one step's host-to-device copies
 * overlap the previous step's computation. Until the step has completed
 * (boute_engine_sync, or a synchronisation of `stream`) its host inputs must
 * stay unchanged and its idx / val must not be read. The second input set is
 * allocated by the first call (B x N x (d + m S) fp32 and the small inputs).
 * boute_engine_sync: waits for every step issued on `stream` and returns the
 * fit status or the first device error.
 * On a non-default stream the step is captured once per argument set (device
 * or host buffers) into a CUDA graph and replayed afterwards; a first call
 * with new pointers therefore must not itself run inside a stream capture.
 * Mode BOUTE_ACQ_NEHVI (m = 2, n <= 128, 1 <= S <= 1024): the noisy
 * acquisition of Sec. 5.2 (see boute_gp_set_insample): after the fit the
 * in-sample draws, then the joint posterior, each draw's front and the
 * draws' hypervolume improvements; eps as for MC_HVI. The engine's S x n
 * in-sample normals per objective come from the generator of
 * boute_base_normals: for seed s (0 at creation, then that of
 * boute_engine_set_normals) they are boute_base_normals(s ^
 * 0x6a09e667f3bcc909, B, m*S, 1, n) read as B x m x S x n. In stage timing
 * the in-sample preparation counts in the fit stage (live) or the front
 * stage (serial), the draws' fronts in the acquisition stage. */
typedef struct boute_engine boute_engine;
int boute_engine_create(int B, int n, int d, int m, long long N, int mode, int S, int k,
                        boute_engine **out);
int boute_engine_step(boute_engine *e, const double *X, const double *Y,
                      const double *lengthscale, const double *outputscale,
                      const double *noise, const double *ref, const float *Xc, const float *eps,
                      long long *idx, float *val, void *stream);
int boute_engine_step_async(boute_engine *e, const double *X, const double *Y,
                            const double *lengthscale, const double *outputscale,
                            const double *noise, const double *ref, const float *Xc,
                            const float *eps, long long *idx, float *val, void *stream);
int boute_engine_step_host(boute_engine *e, const double *X, const double *Y,
                           const double *lengthscale, const double *outputscale,
                           const double *noise, const double *ref, const float *Xc,
                           const float *eps, long long *idx, float *val, void *stream);
int boute_engine_step_host_async(boute_engine *e, const double *X, const double *Y,
                                 const double *lengthscale, const double *outputscale,
                                 const double *noise, const double *ref, const float *Xc,
                                 const float *eps, long long *idx, float *val, void *stream);
int boute_engine_sync(boute_engine *e, void *stream);
/* Copies the last step's per-candidate results into caller buffers (device
 * pointers; any may be NULL): acq B x N, mean and var B x m x N (fp32). */
int boute_engine_scores(const boute_engine *e, float *acq, float *mean, float *var, void *stream);
/* Stage timing on the engine's stream. on = 1 (serialised): every step
 * records a CUDA event at each stage boundary (fit, front = standardise +
 * Pareto front + boxes, posterior, acquisition, top-k) and runs the front
 * stage after the fit on the step's stream instead of beside it, with K*
 * built inside the posterior, so that the stages add up. on = 2 (live): the
 * step keeps its normal concurrent schedule and records events only on the
 * step's stream: "fit" is then everything before the posterior starts (set-up,
 * fit, and any wait for K* built beside it), "front" is 0 (it runs beside the
 * fit), and posterior, acquisition and top-k are the three launches of the
 * scoring pass (top-k is 0 where the acquisition kernel selects). on = 0
 * disables timing. boute_engine_stage_times waits for the last timed step
 * and writes its 5 stage durations in milliseconds (count >= 5). */
int boute_engine_set_timing(boute_engine *e, int on);
int boute_engine_stage_times(boute_engine *e, float *ms, int count);
/* Kernels one boute_engine_step launches. */
int boute_engine_launches_per_step(const boute_engine *e);
/* Constrained acquisition for the engine's later steps (Sec. 5.2,
 * "Constrained qNEHVI"): cons is a HOST array of B x m fp64 thresholds on the
 * standardised, minimised outcomes (the units of the steps' ref), copied into
 * the engine (a NaN threshold is INVALID_ARG); the steps' acquisition becomes
 * E[HVI 1[Y <= cons]] (see boute_acq_ehvi, boute_acq_mc_hvi). cons = NULL
 * returns to the unconstrained acquisition. Waits for all work on the device
 * first (no step may be running); the engine's cached step graphs are rebuilt
 * on the next step when constraints are switched on or off. */
int boute_engine_set_constraints(boute_engine *e, const double *cons);
/* Outcome transforms for the engine's later steps (see boute_standardize):
 * codes is a HOST array of m codes, or NULL for none. The steps' raw outcomes
 * Y are transformed before they are standardised, for the fit and the front
 * alike. Waits for all work on the device when the codes change. */
int boute_engine_set_outcome_transforms(boute_engine *e, const int *codes);
/* The composite kernel for the engine's later steps (see boute_gp_set_kernel;
 * params is a HOST array, NULL restores the Matern-5/2 kernel). */
int boute_engine_set_kernel(boute_engine *e, int d_tau, const double *params);
/* Monte-Carlo engines: draws the engine's own base normals from `seed`
 * (boute_base_normals) into a resident buffer; later steps whose eps is NULL
 * use them (and the host-input steps copy no normals). Synchronous. */
int boute_engine_set_normals(boute_engine *e, unsigned long long seed);
/* A growing data set (Sec. 3.1 loop: one observation is added per
 * iteration): later steps use n observations, 1 <= n <= the n the engine was
 * created with, which fixes every buffer's size; the steps' X and Y then hold
 * n rows. The GP's posterior layout is re-planned for n and the cached step
 * graphs are dropped (the next step on a stream captures a new one); no
 * buffer is allocated, except the in-kernel selection's scratch of
 * 2-objective Monte-Carlo engines when it must grow. Waits for all work on
 * the device. Errors: BOUTE_ERR_INVALID_ARG for n out of range (the engine is
 * unchanged), BOUTE_ERR_OOM / BOUTE_ERR_CUDA (the engine stays usable at
 * n, selecting with the separate top-k kernel). */
int boute_engine_set_n(boute_engine *e, int n);
/* The acquisition optimised over the decision space from the engine's last
 * step (Sec. 5.2 step (ii)): boute_acq_optimize on the engine's fit and the
 * observed front of that step (mode BOUTE_ACQ_MC_HVI, m = 2, the Matern-5/2
 * kernel; otherwise BOUTE_ERR_UNSUPPORTED). Arguments as for
 * boute_acq_optimize (device pointers; X0, X B x P x d). */
int boute_engine_optimize(boute_engine *e, const float *eps, int S, const float *X0, int P,
                          const float *xlo, const float *xhi, int steps, float lr, float *X,
                          float *acq, float *grad, void *stream);
void boute_engine_free(boute_engine *e);

/* ---- the optimisation loop ------------------------------------------------------
 * Sec. 5.2 "Overall MOBO workflow" (i)-(iii), on one problem over a fixed
 * candidate pool: each iteration (i) takes the n observations so far and,
 * when learn_iters > 0, learns the hyperparameters by learn_iters Adam steps
 * from the current ones (boute_gp_learn, one restart; an objective whose
 * kernel matrix is not positive definite keeps its hyperparameters);
 * (ii) scores the pool with the engine (boute_engine_step, k = 1) and
 * (iii) evaluates the best candidate with `f` and adds it to X, Y. It stops
 * when n reaches max_evals or when the observed Pareto set (the observations
 * not dominated after the outcome transforms) has stayed the same for
 * `patience` consecutive iterations (Sec. 7 counts the algorithm converged
 * when the solution is stable for more than 20 consecutive iterations).
 *   f: returns 0 and writes y (m outcomes, raw: before transforms) for x
 *      (d features); a nonzero return stops the loop with INVALID_ARG.
 *   cand: HOST N x d fp32 pool; eps: HOST N x m x S fp32 base normals
 *      (mode BOUTE_ACQ_MC_HVI, reused every iteration), or NULL: the
 *      engine's own normals drawn from cfg->seed (the same every iteration);
 *   ref: m reference point (standardised units); transforms: m codes or
 *      NULL; cons: m thresholds or NULL (the constrained acquisition);
 *   d_tau, kc: the composite kernel (boute_gp_set_kernel's parameters of one
 *      problem, HOST m x (3 + d - d_tau), updated in place when learning:
 *      s2_c, s2_x and beta are learned, the preference entries held), or
 *      kc = NULL for the Matern-5/2 kernel;
 *   ls (m x d), s2 (m), noise (m): HOST hyperparameters, updated in place
 *      when learning;
 *   X (max_evals x d), Y (max_evals x m): HOST, the first n0 rows given;
 *   sel (out, max_evals - n0): the candidate index chosen per iteration
 *      (with refinement: the start whose end point was evaluated);
 *   theta_hist (out, optional, (max_evals - n0) x m x P): the parameters
 *      each iteration scored with (P = d + 2, or d + 5 with the composite
 *      kernel, as for boute_gp_learn / boute_gp_learn_k);
 *   n_out: observations at the end; converged: 1 if the stability test
 *      stopped the loop.
 * Synchronous; allocates its device buffers and one engine for the whole run
 * (created for the largest data set, boute_engine_set_n every iteration). */
typedef int (*boute_objective_fn)(const double *x, int d, double *y, int m, void *user);
typedef struct {
  int mode;         /* BOUTE_ACQ_EHVI2D or BOUTE_ACQ_MC_HVI */
  int S;            /* Monte-Carlo samples (BOUTE_ACQ_MC_HVI) */
  int max_evals;    /* observations at which the loop stops */
  int patience;     /* consecutive iterations of an unchanged Pareto set */
  int learn_iters;  /* Adam steps per iteration; 0 keeps the hyperparameters */
  double learn_lr;  /* Adam step size */
  unsigned long long seed;  /* base normals when eps is NULL (boute_engine_set_normals) */
  /* optional: the acquisition optimised over the decision space (Sec. 5.2
   * step (ii)): from the pool's best refine_starts candidates, refine_steps
   * steps of boute_engine_optimize (step size refine_lr, bounds [0, 1]^d,
   * shared normals boute_base_normals(seed ^ 0xbb67ae8584caa73b, 1, 1, 2, S));
   * the loop then evaluates the best end point (mode BOUTE_ACQ_MC_HVI, m = 2,
   * the Matern-5/2 kernel). refine_steps = 0: the pool's best, as above. */
  int refine_starts, refine_steps;
  double refine_lr;
} boute_mobo_config;
int boute_mobo_run(const boute_mobo_config *cfg, int d, int m, const float *cand, long long N,
                   const float *eps, const double *ref, const int *transforms,
                   const double *cons, int d_tau, double *kc, double *ls, double *s2,
                   double *noise, double *X, double *Y, int n0, boute_objective_fn f, void *user,
                   long long *sel, double *theta_hist, int *n_out, int *converged);

#ifdef __cplusplus
}
#endif
#endif
