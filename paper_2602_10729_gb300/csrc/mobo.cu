// The optimisation loop around the scoring step (Sec. 5.2, "Overall MOBO
// workflow" (i)-(iii)): fit the surrogates (optionally learning their
// hyperparameters), score a candidate pool with the acquisition, evaluate the
// best candidate, add the observation and repeat until the observed Pareto
// set has stayed the same for a number of consecutive iterations (Sec. 7: the
// paper counts the algorithm converged when the solution is stable for more
// than 20 consecutive iterations) or the evaluation budget is spent.
//
// Host code on top of the library's own entry points: every iteration's
// arithmetic runs in the engine's kernels (and the learner's); the loop keeps
// the observations, calls the objective and tests for convergence.
#include <cuda_runtime.h>
#include <math.h>

#include <cstring>
#include <vector>

#include "boute.h"
#include "internal.h"

namespace {

// The outcome transform of one objective (the codes of boute_standardize).
double transformed(double y, int code) {
  double v = y;
  if ((code & 3) == 1) v = log(y);
  else if ((code & 3) == 2) v = log(y / (1.0 - y));
  return (code & 4) ? -v : v;
}

// Indices of the observations not dominated by another (all objectives
// minimised after the transforms); exact duplicates keep the first.
std::vector<int> pareto_set(const double *Y, int n, int m, const int *codes) {
  std::vector<double> z((size_t)n * m);
  for (int i = 0; i < n; ++i)
    for (int t = 0; t < m; ++t) z[(size_t)i * m + t] = transformed(Y[(size_t)i * m + t], codes ? codes[t] : 0);
  std::vector<int> keep;
  for (int i = 0; i < n; ++i) {
    bool dominated = false;
    for (int j = 0; j < n && !dominated; ++j) {
      if (j == i) continue;
      bool le = true, lt = false, eq = true;
      for (int t = 0; t < m; ++t) {
        const double a = z[(size_t)j * m + t], b = z[(size_t)i * m + t];
        le = le && a <= b;
        lt = lt || a < b;
        eq = eq && a == b;
      }
      dominated = (le && lt) || (eq && j < i);
    }
    if (!dominated) keep.push_back(i);
  }
  return keep;
}

template <class T>
int dmalloc(T **p, size_t count) {
  if (cudaMalloc((void **)p, count * sizeof(T) + 16) != cudaSuccess) {
    cudaGetLastError();
    return BOUTE_ERR_OOM;
  }
  return BOUTE_OK;
}

int copy_in(void *dst, const void *src, size_t bytes) {
  return cudaMemcpy(dst, src, bytes, cudaMemcpyHostToDevice) == cudaSuccess ? BOUTE_OK
                                                                            : BOUTE_ERR_CUDA;
}

}  // namespace

extern "C" int boute_mobo_run(const boute_mobo_config *cfg, int d, int m, const float *cand,
                              long long N, const float *eps, const double *ref,
                              const int *transforms, const double *cons, int d_tau, double *kc,
                              double *ls, double *s2, double *noise, double *X, double *Y, int n0,
                              boute_objective_fn f, void *user, long long *sel,
                              double *theta_hist, int *n_out, int *converged) {
  BOUTE_TRACE();
  if (!cfg || !cand || !ref || !ls || !s2 || !noise || !X || !Y || !f || !sel || !n_out ||
      !converged || d < 1 || m < 2 || N < 1 || n0 < 1 || cfg->max_evals < n0 ||
      cfg->patience < 1 || cfg->learn_iters < 0)
    return BOUTE_ERR_INVALID_ARG;
  if (cfg->mode != BOUTE_ACQ_EHVI2D && cfg->S < 1) return BOUTE_ERR_INVALID_ARG;
  if (kc && (d_tau < 0 || d_tau > d)) return BOUTE_ERR_INVALID_ARG;
  // refinement of the pool's best by gradient ascent (optional)
  const bool refine = cfg->refine_steps > 0;
  if (refine && (cfg->refine_starts < 1 || cfg->refine_starts > 1024 ||
                 (long long)cfg->refine_starts > N || !(cfg->refine_lr > 0.0)))
    return BOUTE_ERR_INVALID_ARG;
  if (refine && (cfg->mode != BOUTE_ACQ_MC_HVI || m != 2 || kc)) return BOUTE_ERR_UNSUPPORTED;
  const int KS = refine ? cfg->refine_starts : 1;  // candidates selected per iteration
  // the composite kernel (kc: m x (3 + dc) [s2_c, s2_x, beta, s...]) adds
  // (log s2_c, log s2_x, beta) to the learned parameters
  const int dc = d - d_tau, KC = 3 + dc;
  const int nmax = cfg->max_evals, P = d + (kc ? 5 : 2),
            S = cfg->mode != BOUTE_ACQ_EHVI2D ? cfg->S : 0;
  *n_out = n0;
  *converged = 0;
  double *dX = nullptr, *dY = nullptr, *dYs = nullptr, *dls = nullptr, *ds2 = nullptr,
         *dnz = nullptr, *dref = nullptr, *dth0 = nullptr, *dth = nullptr, *dmll = nullptr,
         *dpref = nullptr;
  float *dXc = nullptr, *deps = nullptr, *dval = nullptr;
  long long *didx = nullptr;
  int r = BOUTE_OK;
  r |= dmalloc(&dX, (size_t)nmax * d);
  r |= dmalloc(&dY, (size_t)nmax * m);
  r |= dmalloc(&dYs, (size_t)nmax * m);
  r |= dmalloc(&dls, (size_t)m * d);
  r |= dmalloc(&ds2, (size_t)m);
  r |= dmalloc(&dnz, (size_t)m);
  r |= dmalloc(&dref, (size_t)m);
  r |= dmalloc(&dth0, (size_t)m * P);
  r |= dmalloc(&dth, (size_t)m * P);
  r |= dmalloc(&dmll, (size_t)m);
  if (kc) r |= dmalloc(&dpref, (size_t)m * dc);
  r |= dmalloc(&dXc, (size_t)N * d);
  if (S && eps) r |= dmalloc(&deps, (size_t)N * m * S);
  r |= dmalloc(&didx, (size_t)KS);
  r |= dmalloc(&dval, (size_t)KS);
  // refinement: start and end points, their values, shared normals, bounds
  float *dX0 = nullptr, *dXo = nullptr, *dacq = nullptr, *deps_r = nullptr, *dlo = nullptr,
        *dhi = nullptr;
  if (refine) {
    r |= dmalloc(&dX0, (size_t)KS * d);
    r |= dmalloc(&dXo, (size_t)KS * d);
    r |= dmalloc(&dacq, (size_t)KS);
    r |= dmalloc(&deps_r, (size_t)2 * S);
    r |= dmalloc(&dlo, (size_t)d);
    r |= dmalloc(&dhi, (size_t)d);
    if (!r) r = boute_base_normals(cfg->seed ^ 0xbb67ae8584caa73bull, 1, 1, 2, S, deps_r, nullptr);
    std::vector<float> zo((size_t)d, 0.f), on((size_t)d, 1.f);
    if (!r) r = copy_in(dlo, zo.data(), sizeof(float) * d);
    if (!r) r = copy_in(dhi, on.data(), sizeof(float) * d);
  }
  if (!r) r = copy_in(dXc, cand, sizeof(float) * N * d);
  if (!r && S && eps) r = copy_in(deps, eps, sizeof(float) * N * m * S);
  if (!r) r = copy_in(dref, ref, sizeof(double) * m);
  if (!r && kc) {  // the preference entries (held fixed)
    std::vector<double> pr((size_t)m * dc);
    for (int t = 0; t < m; ++t)
      for (int k = 0; k < dc; ++k) pr[(size_t)t * dc + k] = kc[(size_t)t * KC + 3 + k];
    r = copy_in(dpref, pr.data(), sizeof(double) * m * dc);
  }
  // one engine for the whole loop, sized for its largest data set (n grows
  // by one per iteration up to nmax - 1 before the last selection)
  boute_engine *e = nullptr;
  if (!r && n0 < nmax) r = boute_engine_create(1, nmax - 1, d, m, N, cfg->mode, S, KS, &e);
  if (!r && transforms) r = boute_engine_set_outcome_transforms(e, transforms);
  if (!r && cons) r = boute_engine_set_constraints(e, cons);
  if (!r && S && !eps) r = boute_engine_set_normals(e, cfg->seed);  // eps null: own normals
  std::vector<int> front = pareto_set(Y, n0, m, transforms);
  int n = n0, stable = 0, it = 0;
  std::vector<double> th((size_t)m * P);
  while (!r && n < nmax) {
    // (i) surrogates: the observations so far, hyperparameters learned from
    // the current ones (warm start) when asked
    r = copy_in(dX, X, sizeof(double) * n * d);
    if (!r) r = copy_in(dY, Y, sizeof(double) * n * m);
    for (int t = 0; t < m; ++t) {
      for (int q = 0; q < d; ++q) th[(size_t)t * P + q] = log(ls[(size_t)t * d + q]);
      th[(size_t)t * P + d] = log(s2[t]);
      th[(size_t)t * P + d + 1] = log(noise[t]);
      if (kc) {
        th[(size_t)t * P + d + 2] = log(kc[(size_t)t * KC]);
        th[(size_t)t * P + d + 3] = log(kc[(size_t)t * KC + 1]);
        th[(size_t)t * P + d + 4] = kc[(size_t)t * KC + 2];
      }
    }
    if (!r && cfg->learn_iters > 0) {
      r = boute_standardize(dY, 1, n, m, transforms, dYs, nullptr);
      if (!r) r = copy_in(dth0, th.data(), sizeof(double) * m * P);
      if (!r)
        r = kc ? boute_gp_learn_k(dX, dYs, 1, n, d, m, d_tau, dpref, dth0, 1, cfg->learn_iters,
                                  cfg->learn_lr, dth, dmll, nullptr, nullptr)
               : boute_gp_learn(dX, dYs, 1, n, d, m, dth0, 1, cfg->learn_iters, cfg->learn_lr,
                                dth, dmll, nullptr, nullptr);
      std::vector<double> thn((size_t)m * P), mll(m);
      if (!r && (cudaMemcpy(thn.data(), dth, sizeof(double) * m * P, cudaMemcpyDeviceToHost) !=
                     cudaSuccess ||
                 cudaMemcpy(mll.data(), dmll, sizeof(double) * m, cudaMemcpyDeviceToHost) !=
                     cudaSuccess))
        r = BOUTE_ERR_CUDA;
      for (int t = 0; !r && t < m; ++t) {
        if (!(mll[t] == mll[t])) continue;  // not positive definite: keep the last ones
        std::memcpy(&th[(size_t)t * P], &thn[(size_t)t * P], sizeof(double) * P);
        for (int q = 0; q < d; ++q) ls[(size_t)t * d + q] = exp(th[(size_t)t * P + q]);
        s2[t] = exp(th[(size_t)t * P + d]);
        noise[t] = exp(th[(size_t)t * P + d + 1]);
        if (kc) {
          kc[(size_t)t * KC] = exp(th[(size_t)t * P + d + 2]);
          kc[(size_t)t * KC + 1] = exp(th[(size_t)t * P + d + 3]);
          kc[(size_t)t * KC + 2] = th[(size_t)t * P + d + 4];
        }
      }
    }
    if (theta_hist) std::memcpy(theta_hist + (size_t)it * m * P, th.data(), sizeof(double) * m * P);
    if (!r) r = copy_in(dls, ls, sizeof(double) * m * d);
    if (!r) r = copy_in(ds2, s2, sizeof(double) * m);
    if (!r) r = copy_in(dnz, noise, sizeof(double) * m);
    // (ii) the acquisition over the pool and its best candidate
    if (!r) r = boute_engine_set_n(e, n);
    if (!r && kc) r = boute_engine_set_kernel(e, d_tau, kc);
    if (!r) r = boute_engine_step(e, dX, dY, dls, ds2, dnz, dref, dXc, deps, didx, dval, nullptr);
    std::vector<long long> picks((size_t)KS, -1);
    if (!r && cudaMemcpy(picks.data(), didx, sizeof(long long) * KS, cudaMemcpyDeviceToHost) !=
                  cudaSuccess)
      r = BOUTE_ERR_CUDA;
    if (r) break;
    long long pick = picks[0];
    double *xn = X + (size_t)n * d, *yn = Y + (size_t)n * m;
    for (int q = 0; q < d; ++q) xn[q] = (double)cand[(size_t)pick * d + q];
    if (refine) {  // gradient ascent from the pool's best KS; the best end point
      std::vector<float> x0((size_t)KS * d), xo((size_t)KS * d), ao((size_t)KS);
      for (int p = 0; p < KS; ++p)
        for (int q = 0; q < d; ++q) x0[(size_t)p * d + q] = cand[(size_t)picks[p] * d + q];
      r = copy_in(dX0, x0.data(), sizeof(float) * KS * d);
      if (!r)
        r = boute_engine_optimize(e, deps_r, S, dX0, KS, dlo, dhi, cfg->refine_steps,
                                  (float)cfg->refine_lr, dXo, dacq, nullptr, nullptr);
      if (!r && (cudaMemcpy(xo.data(), dXo, sizeof(float) * KS * d, cudaMemcpyDeviceToHost) !=
                     cudaSuccess ||
                 cudaMemcpy(ao.data(), dacq, sizeof(float) * KS, cudaMemcpyDeviceToHost) !=
                     cudaSuccess))
        r = BOUTE_ERR_CUDA;
      if (r) break;
      int best = 0;
      for (int p = 1; p < KS; ++p)
        if (ao[p] > ao[best]) best = p;
      pick = picks[best];
      for (int q = 0; q < d; ++q) xn[q] = (double)xo[(size_t)best * d + q];
    }
    // (iii) evaluate it and add the observation
    if (f(xn, d, yn, m, user) != 0) {
      r = BOUTE_ERR_INVALID_ARG;
      break;
    }
    sel[it++] = pick;
    ++n;
    // convergence: the observed Pareto set unchanged for `patience` iterations
    std::vector<int> fr = pareto_set(Y, n, m, transforms);
    stable = fr == front ? stable + 1 : 0;
    front.swap(fr);
    if (stable >= cfg->patience) {
      *converged = 1;
      break;
    }
  }
  *n_out = n;
  boute_engine_free(e);
  void *bufs[] = {dX,   dY,  dYs,  dls, ds2,  dnz,  dref,   dth0, dth, dmll,
                  dXc,  deps, didx, dval, dpref, dX0, dXo, dacq, deps_r, dlo, dhi};
  for (void *p : bufs) cudaFree(p);
  return r;
}
