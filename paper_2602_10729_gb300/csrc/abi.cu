// The C ABI of libboute (declared in include/boute.h): argument validation,
// handle and engine ownership, and the launch sequence of one scoring step.
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "internal.h"

namespace boute {

static std::atomic<unsigned long long> g_launches{0};
void count_launch(int k) { g_launches.fetch_add((unsigned long long)k); }
// Launches recorded while capturing a graph ran nothing; they count when the
// graph is launched.
static void g_launches_adjust(int captured) {
  g_launches.fetch_sub((unsigned long long)captured);
}
unsigned long long launch_count() { return g_launches.load(); }

int last_launch_status() {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) return BOUTE_OK;
  if (e == cudaErrorMemoryAllocation) return BOUTE_ERR_OOM;
  std::fprintf(stderr, "libboute: %s\n", cudaGetErrorString(e));
  return BOUTE_ERR_CUDA;
}

// The kernels are built for sm_103a only: refuse other devices up front (a
// failed device query leaves no error behind for later calls to report).
int device_ok() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return BOUTE_ERR_UNSUPPORTED;
  }
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return (major == 10 && minor == 3) ? BOUTE_OK : BOUTE_ERR_UNSUPPORTED;
}

template <class T>
static int dalloc(T **p, size_t count) {
  *p = nullptr;
  if (count == 0) return BOUTE_OK;
  cudaError_t e = cudaMalloc((void **)p, count * sizeof(T));
  if (e != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return BOUTE_ERR_OOM;
  }
  return BOUTE_OK;
}

static int pad_dims(int d) { return d <= 8 ? 8 : d <= 12 ? 12 : d <= 16 ? 16 : d <= 24 ? 24 : 32; }

static int shape_ok(int B, int n, int d, int m) {
  return B >= 1 && n >= 1 && n <= BOUTE_MAX_N && d >= 1 && d <= BOUTE_MAX_D && m >= 1 &&
         m <= BOUTE_MAX_M;
}

}  // namespace boute

using namespace boute;

struct boute_gp {
  Gp g;
};

// copy streams of a host-input step (the normals are split over all of them)
constexpr int kCopyStreams = 2;

struct boute_engine {
  int B, n, d, m, mode, S, k;
  int ncap;  // the buffers hold up to ncap observations (boute_engine_set_n)
  long long N;
  boute_gp *gp;
  double *X, *Y, *Ys, *ls, *s2, *noise, *ref, *front;
  unsigned char *mask;
  int *P, *K;
  float *lower, *upper, *Xc, *eps, *mean, *var, *acq, *val;
  long long *idx;
  void *scratch;
  // 2-objective Monte-Carlo steps with k <= 32 select in the acquisition
  // kernel: its lists of keys and counters (zero between steps)
  unsigned char *sel;
  size_t sel_bytes;
  bool fuse_sel;
  // K* of the candidates, computed on a second side stream while the fit
  // runs (it needs the fit's set-up, not its results); the posterior then
  // only contracts it. Null when it would take more than kKstarMaxBytes.
  float *kst;
  cudaStream_t side2;
  cudaEvent_t ev_setup, join2;
  int launches;
  int timing;                  // record one CUDA event per stage boundary
  cudaEvent_t ev[8];           // boundaries of the stages of the last step
  int nstage;
  // the step as a CUDA graph, per argument set (two sets: device and host
  // inputs); replay removes the host launch gaps between the kernels
  struct Graph {
    const void *key[12];
    cudaGraphExec_t exec;
    int launches;
  } graphs[3];
  int graph_next, graphs_off;
  // the front stage (standardise, Pareto front, boxes) depends on the raw
  // outcomes only: it runs on a second stream, forked after the fit's set-up
  // (ev_setup) and joined back into the step's stream, beside the GP fit
  cudaStream_t side;
  cudaEvent_t join;
  // host-input steps: candidates and base normals are copied on kCopyStreams
  // copy streams while the fit runs (the normals split evenly over them, so
  // that several copy engines carry them); the step waits for them only where
  // it needs them (posterior, acquisition)
  cudaStream_t cpy[kCopyStreams];
  cudaEvent_t ev_in, ev_xc, ev_eps[kCopyStreams];
  // pipelined host-input steps: a second set of device input buffers (the
  // first is X .. eps above, allocated on first use) so that one step's copies
  // overlap the previous step's computation; in_free[s] marks the end of the
  // last step that read set s
  double *X1, *Y1, *ls1, *s21, *noise1, *ref1;
  float *Xc1, *eps1;
  cudaEvent_t ev_xc1, ev_eps1[kCopyStreams], in_free[2];
  cudaEvent_t ev_small[2];  // the small inputs of set 0 / 1 are in place
  int host_set;
  // constrained acquisition (boute_engine_set_constraints): B x m thresholds,
  // allocated on first use; used while has_cons
  double *cons;
  int has_cons;
  // outcome transforms (boute_engine_set_outcome_transforms): the step first
  // writes the transformed outcomes to Yt, which the fit and the front read
  int tcodes;
  double *Yt;
  // the engine's own base normals (boute_engine_set_normals), used by steps
  // whose eps is null; null until set
  float *gen_eps;
  // noisy acquisition (BOUTE_ACQ_NEHVI): in-sample normals (B x m x S x n,
  // drawn from zseed), in-sample draws, the posterior's shifts (B x m x S x N),
  // and the draws' fronts as strips (B x S x (n + 1) x 4) with their counts
  float *zin, *Yin, *shift, *strips;
  int *counts;
  unsigned long long zseed;
};

namespace boute {
// Key of the in-sample normals of seed s: s ^ kInsampleKey (the first 64
// bits of the fractional part of sqrt(2)), so that they are drawn
// independently of the candidates' normals of the same seed.
constexpr unsigned long long kInsampleKey = 0x6a09e667f3bcc909ull;
static int draw_insample_normals(boute_engine *e, cudaStream_t s) {
  return launch_base_normals(e->zseed ^ kInsampleKey, e->B, (long long)e->m * e->S, 1, e->n,
                             e->zin, s);
}
}  // namespace boute

// Stage order of one step as timed (with timing on, the front stage runs
// after the fit on the step's stream, so the stage times add up).
enum { ST_FIT, ST_FRONT, ST_POSTERIOR, ST_ACQ, ST_TOPK, ST_COUNT };

extern "C" {

const char *boute_status_string(int s) {
  switch (s) {
    case BOUTE_OK: return "ok";
    case BOUTE_ERR_INVALID_ARG: return "invalid argument";
    case BOUTE_ERR_NOT_PD: return "kernel matrix not positive definite";
    case BOUTE_ERR_CUDA: return "CUDA error";
    case BOUTE_ERR_OOM: return "out of device memory";
    case BOUTE_ERR_UNSUPPORTED: return "unsupported device or shape";
    case BOUTE_ERR_TIMEOUT: return "device-side wait timed out";
  }
  return "unknown status";
}

unsigned long long boute_launch_count(void) { return launch_count(); }

// m per-objective transform codes (host, or null = identity) packed 3 bits
// apiece; false for an unknown code
static bool pack_codes(const int *codes, int m, int *packed) {
  *packed = 0;
  if (!codes) return true;
  for (int t = 0; t < m; ++t) {
    const int c = codes[t];
    if (c < 0 || c > 7 || (c & 3) == 3) return false;
    *packed |= c << (3 * t);
  }
  return true;
}

int boute_standardize(const double *Y, int B, int n, int m, const int *transforms, double *Ys,
                      void *stream) {
  BOUTE_TRACE();
  int codes = 0;
  if (!Y || !Ys || B < 1 || n < 1 || m < 1 || m > BOUTE_MAX_M || !pack_codes(transforms, m, &codes))
    return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  return launch_standardize(Y, B, n, m, codes, Ys, (cudaStream_t)stream);
}

int boute_gp_create(int B, int n, int d, int m, boute_gp **out) {
  BOUTE_TRACE();
  if (!out) return BOUTE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!shape_ok(B, n, d, m)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  boute_gp *h = new (std::nothrow) boute_gp();
  if (!h) return BOUTE_ERR_OOM;
  Gp &g = h->g;
  g.B = B; g.n = n; g.d = d; g.m = m; g.DP = pad_dims(d);
  g.ncap = n;
  g.plan = make_post_plan(n);
  const size_t BM = (size_t)B * m;
  int r = BOUTE_OK;
  r |= dalloc(&g.Kh, BM * n * n);
  r |= dalloc(&g.Kl, BM * n * n);
  const size_t np = g.plan.npad;
  r |= dalloc(&g.Aws, BM * np * (np + 1));
  r |= dalloc(&g.Wws, BM * np * (np + 1));
  r |= dalloc(&g.bop, BM * (size_t)g.plan.image_halves);
  g.kcache_chunks = g.kcache_cap = kstar_cache_chunks(g.plan);
  g.kcache_sms = num_sms();
  if (g.kcache_chunks > 0)
    r |= dalloc(&g.kcache, (size_t)g.kcache_sms * g.kcache_chunks * kKstarChunkHalves);
  r |= dalloc(&g.xt, BM * (size_t)g.plan.nxt * xt_chunk_floats(g.DP));
  r |= dalloc(&g.s2f, BM);
  r |= dalloc(&g.status, 1);
  r |= dalloc(&g.fbad, BM);
  if (const size_t tp = fit_tpart_floats((int)np, (int)BM)) r |= dalloc(&g.tpart, tp);
  if (const size_t fv = fit_fvec_floats((int)np, (int)BM)) r |= dalloc(&g.fvec, fv);
  if (r != BOUTE_OK) {
    boute_gp_free(h);
    return BOUTE_ERR_OOM;
  }
  cudaMemset(g.status, 0, sizeof(int));
  // operand images are fully rewritten by every fit; zero them once so that
  // padding never holds stale bits
  cudaMemset(g.bop, 0, BM * (size_t)g.plan.image_halves * sizeof(uint16_t));
  cudaMemset(g.xt, 0, BM * (size_t)g.plan.nxt * xt_chunk_floats(g.DP) * sizeof(float));
  *out = h;
  return BOUTE_OK;
}

int boute_gp_fit(boute_gp *gp, const double *X, const double *Ys, const double *lengthscale,
                 const double *outputscale, const double *noise, void *stream) {
  BOUTE_TRACE();
  if (!gp || !X || !Ys || !lengthscale || !outputscale || !noise) return BOUTE_ERR_INVALID_ARG;
  Gp &g = gp->g;
  const cudaStream_t s = (cudaStream_t)stream;
  if (int r = launch_fit(&g, X, Ys, lengthscale, outputscale, noise, s)) return r;
  if (g.prec != BOUTE_PREC_FP64) return BOUTE_OK;
  const size_t BM = (size_t)g.B * g.m;
  if (cudaMemcpyAsync(g.ls64, lengthscale, BM * g.d * sizeof(double), cudaMemcpyDeviceToDevice,
                      s) != cudaSuccess ||
      cudaMemcpyAsync(g.s2_64, outputscale, BM * sizeof(double), cudaMemcpyDeviceToDevice, s) !=
          cudaSuccess)
    return last_launch_status();
  return launch_fit64(&g, X, Ys, lengthscale, outputscale, noise, s);
}

int boute_gp_set_precision(boute_gp *gp, int prec) {
  BOUTE_TRACE();
  if (!gp || (prec != BOUTE_PREC_FP32 && prec != BOUTE_PREC_FP64)) return BOUTE_ERR_INVALID_ARG;
  Gp &g = gp->g;
  if (prec == BOUTE_PREC_FP64) {
    if (g.n > kFp64MaxN || g.kern || g.plan.S_in > 0) return BOUTE_ERR_UNSUPPORTED;
    if (!g.W64) {
      const size_t BM = (size_t)g.B * g.m;
      int r = dalloc(&g.W64, BM * g.n * g.n);
      r |= dalloc(&g.a64, BM * g.n);
      r |= dalloc(&g.xs64, BM * g.n * g.d);
      r |= dalloc(&g.ls64, BM * g.d);
      r |= dalloc(&g.s2_64, BM);
      if (r != BOUTE_OK) return BOUTE_ERR_OOM;
    }
  }
  g.prec = prec;
  return BOUTE_OK;
}

int boute_gp_posterior_fp64(const boute_gp *gp, const float *Xc, long long N, double *mean,
                            double *var, void *stream) {
  BOUTE_TRACE();
  if (!gp || N < 0 || (N > 0 && (!Xc || !mean || !var))) return BOUTE_ERR_INVALID_ARG;
  if (gp->g.prec != BOUTE_PREC_FP64) return BOUTE_ERR_INVALID_ARG;
  return launch_posterior64(&gp->g, Xc, N, mean, var, (cudaStream_t)stream);
}

// ---- noisy acquisition: in-sample draws -----------------------------------------
int boute_gp_set_insample(boute_gp *gp, int S) {
  BOUTE_TRACE();
  if (!gp || S < 0 || S > kInsMaxS) return BOUTE_ERR_INVALID_ARG;
  Gp &g = gp->g;
  if (S == g.plan.S_in) return BOUTE_OK;
  if (S > 0 && (g.ncap > kInsMaxN || g.prec != BOUTE_PREC_FP32)) return BOUTE_ERR_UNSUPPORTED;
  if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  const size_t BM = (size_t)g.B * g.m;
  const PostPlan cap = make_post_plan(g.ncap, S);
  // new operand images (W's blocks then H^T's and G^T's), zero: fit again
  uint16_t *bop = nullptr;
  if (dalloc(&bop, BM * (size_t)cap.image_halves) != BOUTE_OK) return BOUTE_ERR_OOM;
  float *gws = nullptr, *iws = nullptr;
  if (S > 0 && (dalloc(&gws, BM * (size_t)S * g.ncap) != BOUTE_OK ||
                dalloc(&iws, BM * insample_ws_floats(g.ncap)) != BOUTE_OK)) {
    cudaFree(bop);
    cudaFree(gws);
    return BOUTE_ERR_OOM;
  }
  const int want = kstar_cache_chunks(cap);
  uint16_t *kc = nullptr;
  if (want > g.kcache_cap &&
      dalloc(&kc, (size_t)g.kcache_sms * want * kKstarChunkHalves) != BOUTE_OK) {
    cudaFree(bop);
    cudaFree(gws);
    cudaFree(iws);
    return BOUTE_ERR_OOM;
  }
  if (cudaMemset(bop, 0, BM * (size_t)cap.image_halves * sizeof(uint16_t)) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(bop);
    cudaFree(gws);
    cudaFree(iws);
    cudaFree(kc);
    return BOUTE_ERR_CUDA;
  }
  cudaFree(g.bop);
  g.bop = bop;
  cudaFree(g.gws);
  g.gws = gws;
  cudaFree(g.iws);
  g.iws = iws;
  if (kc) {
    cudaFree(g.kcache);
    g.kcache = kc;
    g.kcache_cap = want;
  }
  g.plan = make_post_plan(g.n, S);
  const int now = kstar_cache_chunks(g.plan);
  g.kcache_chunks = now <= g.kcache_cap ? now : 0;
  return BOUTE_OK;
}

int boute_gp_insample(boute_gp *gp, const double *Ys, const double *outputscale,
                      const double *noise, const float *z, float *Yin, void *stream) {
  BOUTE_TRACE();
  if (!gp || !Ys || !outputscale || !noise || !z || !Yin) return BOUTE_ERR_INVALID_ARG;
  if (gp->g.plan.S_in < 1) return BOUTE_ERR_INVALID_ARG;
  return launch_insample(&gp->g, Ys, outputscale, noise, z, Yin, (cudaStream_t)stream);
}

int boute_gp_posterior_joint(const boute_gp *gp, const float *Xc, long long N, float *mean,
                             float *cvar, float *shift, void *stream) {
  BOUTE_TRACE();
  if (!gp || N < 0 || (N > 0 && (!Xc || !mean || !cvar || !shift))) return BOUTE_ERR_INVALID_ARG;
  if (gp->g.plan.S_in < 1) return BOUTE_ERR_INVALID_ARG;
  if ((long long)gp->g.B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  return launch_posterior_joint(&gp->g, Xc, N, mean, cvar, shift, (cudaStream_t)stream);
}

int boute_insample_fronts(const float *Yin, int B, int n, int S, const double *ref,
                          const double *cons, float *strips, int *counts, void *stream) {
  BOUTE_TRACE();
  if (!Yin || !ref || !strips || !counts || B < 1 || n < 1 || S < 1 || S > kInsMaxS)
    return BOUTE_ERR_INVALID_ARG;
  if (n > kInsMaxN) return BOUTE_ERR_UNSUPPORTED;
  if (int r = device_ok()) return r;
  return launch_insample_fronts(Yin, B, n, S, ref, cons, strips, counts, (cudaStream_t)stream);
}

int boute_acq_nehvi2d(const float *mean, const float *cvar, const float *shift, int B,
                      long long N, int S, const float *eps, long long eps_cand_stride,
                      const float *strips, const int *counts, int n, const double *cons,
                      float *acq, void *stream) {
  BOUTE_TRACE();
  if (B < 1 || N < 0 || S < 1 || S > kInsMaxS || n < 1 || eps_cand_stride < 0 || !strips ||
      !counts || (N > 0 && (!mean || !cvar || !shift || !eps || !acq)))
    return BOUTE_ERR_INVALID_ARG;
  if (n > kInsMaxN) return BOUTE_ERR_UNSUPPORTED;
  if ((long long)B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  if (N == 0) return BOUTE_OK;
  return launch_nehvi2(mean, cvar, shift, B, N, S, eps, eps_cand_stride, strips, counts, n, cons,
                       acq, (cudaStream_t)stream);
}

int boute_gp_status(boute_gp *gp, void *stream) {
  BOUTE_TRACE();
  if (!gp) return BOUTE_ERR_INVALID_ARG;
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return last_launch_status();
  int st = 0;
  if (cudaMemcpy(&st, gp->g.status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return last_launch_status();
  cudaMemset(gp->g.status, 0, sizeof(int));
  return st;
}

void boute_gp_free(boute_gp *gp) {
  BOUTE_TRACE();
  if (!gp) return;
  Gp &g = gp->g;
  cudaFree(g.Kh); cudaFree(g.Kl); cudaFree(g.Aws); cudaFree(g.Wws); cudaFree(g.bop); cudaFree(g.xt);
  cudaFree(g.s2f); cudaFree(g.status); cudaFree(g.kpar); cudaFree(g.kcache); cudaFree(g.fbad);
  cudaFree(g.tpart); cudaFree(g.fvec);
  cudaFree(g.W64); cudaFree(g.a64); cudaFree(g.xs64); cudaFree(g.ls64); cudaFree(g.s2_64);
  cudaFree(g.gws);
  cudaFree(g.iws);
  delete gp;
}

int boute_gp_learn(const double *X, const double *Ys, int B, int n, int d, int m,
                   const double *theta0, int R, int iters, double lr, double *theta,
                   double *mll, double *grad, void *stream) {
  BOUTE_TRACE();
  if (!X || !Ys || !theta0 || !theta || !mll || !shape_ok(B, n, d, m) || R < 1 || iters < 0 ||
      !(lr >= 0.0))
    return BOUTE_ERR_INVALID_ARG;
  if ((long long)B * m * R > (1ll << 30)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  return launch_learn(X, Ys, B, n, d, m, theta0, R, iters, lr, theta, mll, grad, d, nullptr,
                      (cudaStream_t)stream);
}

int boute_gp_learn_k(const double *X, const double *Ys, int B, int n, int d, int m, int d_tau,
                     const double *pref, const double *theta0, int R, int iters, double lr,
                     double *theta, double *mll, double *grad, void *stream) {
  BOUTE_TRACE();
  if (!X || !Ys || !pref || !theta0 || !theta || !mll || !shape_ok(B, n, d, m) || R < 1 ||
      iters < 0 || !(lr >= 0.0) || d_tau < 0 || d_tau > d)
    return BOUTE_ERR_INVALID_ARG;
  if ((long long)B * m * R > (1ll << 30)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  return launch_learn(X, Ys, B, n, d, m, theta0, R, iters, lr, theta, mll, grad, d_tau, pref,
                      (cudaStream_t)stream);
}

int boute_gp_set_kernel(boute_gp *gp, int d_tau, const double *params) {
  BOUTE_TRACE();
  if (!gp) return BOUTE_ERR_INVALID_ARG;
  Gp &g = gp->g;
  if (!params) {
    g.kern = 0;
    return BOUTE_OK;
  }
  if (g.prec == BOUTE_PREC_FP64) return BOUTE_ERR_UNSUPPORTED;  // (Matern-5/2 only)
  if (d_tau < 0 || d_tau > g.d) return BOUTE_ERR_INVALID_ARG;
  const int BM = g.B * g.m, dc = g.d - d_tau, in = 3 + dc, out = 3 + g.d;
  std::vector<double> h((size_t)BM * out, 0.0);
  for (int bt = 0; bt < BM; ++bt) {
    const double *p = params + (size_t)bt * in;
    double *q = h.data() + (size_t)bt * out;
    q[0] = p[0];
    q[1] = p[1];
    q[2] = p[2];
    for (int k = 0; k < dc; ++k) q[3 + d_tau + k] = p[3 + k];
  }
  // no fit of this handle may be reading the parameters while they change
  if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  if (!g.kpar && dalloc(&g.kpar, h.size()) != BOUTE_OK) return BOUTE_ERR_OOM;
  if (cudaMemcpy(g.kpar, h.data(), h.size() * sizeof(double), cudaMemcpyHostToDevice) !=
      cudaSuccess)
    return last_launch_status();
  g.kern = 1;
  g.dtau = d_tau;
  return BOUTE_OK;
}

int boute_gp_posterior(const boute_gp *gp, const float *Xc, long long N, float *mean, float *var,
                       void *stream) {
  BOUTE_TRACE();
  if (!gp || N < 0 || (N > 0 && (!Xc || !mean || !var))) return BOUTE_ERR_INVALID_ARG;
  if ((long long)gp->g.B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  return launch_posterior(&gp->g, Xc, N, mean, var, (cudaStream_t)stream);
}

int boute_pareto_front(const double *Ys, int B, int n, int m, const double *ref,
                       unsigned char *mask, double *front, int *P, void *stream) {
  BOUTE_TRACE();
  if (!Ys || !ref || !mask || !front || !P || !shape_ok(B, n, 1, m)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  return launch_pareto(Ys, B, n, m, ref, mask, front, P, (cudaStream_t)stream);
}

int boute_box_decompose(const double *front, const int *P, int B, int n, int m, const double *ref,
                        float *lower, float *upper, int *K, void *stream) {
  BOUTE_TRACE();
  if (!front || !P || !ref || !lower || !upper || !K || !shape_ok(B, n, 1, m))
    return BOUTE_ERR_INVALID_ARG;
  if (m < 2 || m > 3) return BOUTE_ERR_UNSUPPORTED;
  if (int r = device_ok()) return r;
  return launch_boxes(front, P, B, n, m, ref, lower, upper, K, (cudaStream_t)stream);
}

int boute_acq_ehvi(const float *mean, const float *var, int B, long long N, const double *front,
                   const int *P, int n, const double *ref, const double *cons, float *acq,
                   void *stream) {
  BOUTE_TRACE();
  if (B < 1 || N < 0 || n < 1 || n > BOUTE_MAX_N || !front || !P || !ref ||
      (N > 0 && (!mean || !var || !acq)))
    return BOUTE_ERR_INVALID_ARG;
  if ((long long)B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  return launch_ehvi(mean, var, B, N, front, P, n, ref, cons, acq, (cudaStream_t)stream);
}

int boute_acq_mc_hvi(const float *mean, const float *var, int B, long long N, int m,
                     const float *lower, const float *upper, const int *K, int box_cap,
                     const float *eps, int S, long long eps_cand_stride, const double *cons,
                     float *acq, void *stream) {
  BOUTE_TRACE();
  if (B < 1 || N < 0 || S < 1 || box_cap < 1 || eps_cand_stride < 0 || !lower || !upper || !K ||
      (N > 0 && (!mean || !var || !acq || !eps)))
    return BOUTE_ERR_INVALID_ARG;
  if (m < 2 || m > 3) return BOUTE_ERR_UNSUPPORTED;
  if ((long long)B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  if ((size_t)box_cap * m * 2 * sizeof(float) > 200 * 1024) return BOUTE_ERR_UNSUPPORTED;
  if (int r = device_ok()) return r;
  return launch_mchvi(mean, var, B, N, m, lower, upper, K, box_cap, eps, S, eps_cand_stride, cons,
                      acq, (cudaStream_t)stream);
}

int boute_select_topk(const float *acq, int B, long long N, int k, long long *idx, float *val,
                      void *stream) {
  BOUTE_TRACE();
  if (!acq || !idx || !val || B < 1 || N < 1 || k < 1 || k > 1024 || k > N)
    return BOUTE_ERR_INVALID_ARG;
  if ((long long)B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  cudaStream_t s = (cudaStream_t)stream;
  void *scratch = nullptr;
  if (cudaMallocAsync(&scratch, topk_scratch_bytes(B, N, k), s) != cudaSuccess) {
    cudaGetLastError();
    return BOUTE_ERR_OOM;
  }
  int r = launch_topk(acq, B, N, k, idx, val, scratch, s);
  cudaFreeAsync(scratch, s);
  return r;
}

// ---- engine -------------------------------------------------------------------
void boute_engine_free(boute_engine *e) {
  BOUTE_TRACE();
  if (!e) return;
  boute_gp_free(e->gp);
  if (e->ev[0])
    for (int i = 0; i <= ST_COUNT; ++i) cudaEventDestroy(e->ev[i]);
  for (auto &g : e->graphs)
    if (g.exec) cudaGraphExecDestroy(g.exec);
  if (e->join) cudaEventDestroy(e->join);
  if (e->side) cudaStreamDestroy(e->side);
  for (cudaEvent_t ev : {e->ev_in, e->ev_xc, e->ev_setup, e->join2, e->ev_xc1, e->in_free[0],
                         e->in_free[1], e->ev_small[0], e->ev_small[1]})
    if (ev) cudaEventDestroy(ev);
  for (int i = 0; i < kCopyStreams; ++i) {
    if (e->ev_eps[i]) cudaEventDestroy(e->ev_eps[i]);
    if (e->ev_eps1[i]) cudaEventDestroy(e->ev_eps1[i]);
  }
  if (e->side2) cudaStreamDestroy(e->side2);
  for (cudaStream_t c : e->cpy)
    if (c) cudaStreamDestroy(c);
  void *ptrs[] = {e->X, e->Y, e->Ys, e->ls, e->s2, e->noise, e->ref, e->front, e->mask, e->P,
                  e->K, e->lower, e->upper, e->Xc, e->eps, e->mean, e->var, e->acq, e->val,
                  e->idx, e->scratch, e->sel, e->kst, e->X1, e->Y1, e->ls1, e->s21,
                  e->noise1, e->ref1, e->Xc1, e->eps1, e->cons, e->Yt, e->gen_eps,
                  e->zin,    e->Yin,  e->shift, e->strips, e->counts};
  for (void *p : ptrs) cudaFree(p);
  delete e;
}

// Largest K* buffer an engine keeps (it lets the posterior's K* be computed
// beside the fit); larger workloads build K* inside the posterior.
constexpr size_t kKstarMaxBytes = size_t(512) << 20;

// The selection runs inside the acquisition kernel for 2-objective
// Monte-Carlo steps with k <= 32 (not in stage-timing mode, which times the
// selection as a stage of its own).
static bool engine_fuses_selection(const boute_engine *e) {
  return e->mode == BOUTE_ACQ_MC_HVI && e->m == 2 && e->k <= 32 &&
         mchvi2_select_grid_x(e->B, e->N, 2 * e->n + 2) <= 32 * 32;
}

int boute_engine_create(int B, int n, int d, int m, long long N, int mode, int S, int k,
                        boute_engine **out) {
  BOUTE_TRACE();
  if (!out) return BOUTE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!shape_ok(B, n, d, m) || N < 1 || k < 1 || k > 1024 || k > N) return BOUTE_ERR_INVALID_ARG;
  if ((long long)B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  if (mode == BOUTE_ACQ_EHVI2D && m != 2) return BOUTE_ERR_INVALID_ARG;
  if (mode == BOUTE_ACQ_MC_HVI && (m < 2 || m > 3 || S < 1)) return BOUTE_ERR_INVALID_ARG;
  if (mode == BOUTE_ACQ_NEHVI && (m != 2 || S < 1 || S > kInsMaxS)) return BOUTE_ERR_INVALID_ARG;
  if (mode != BOUTE_ACQ_EHVI2D && mode != BOUTE_ACQ_MC_HVI && mode != BOUTE_ACQ_NEHVI)
    return BOUTE_ERR_INVALID_ARG;
  if (mode == BOUTE_ACQ_NEHVI && n > kInsMaxN) return BOUTE_ERR_UNSUPPORTED;
  if (int r = device_ok()) return r;
  boute_engine *e = new (std::nothrow) boute_engine();
  if (!e) return BOUTE_ERR_OOM;
  std::memset(e, 0, sizeof(*e));
  e->B = B; e->n = n; e->d = d; e->m = m; e->N = N; e->mode = mode; e->S = S; e->k = k;
  e->ncap = n;
  int r = boute_gp_create(B, n, d, m, &e->gp);
  const size_t Bn = (size_t)B * n, BN = (size_t)B * N, cap = 2 * (size_t)n + 2;
  r |= dalloc(&e->X, Bn * d);
  r |= dalloc(&e->Y, Bn * m);
  r |= dalloc(&e->Ys, Bn * m);
  r |= dalloc(&e->ls, (size_t)B * m * d);
  r |= dalloc(&e->s2, (size_t)B * m);
  r |= dalloc(&e->noise, (size_t)B * m);
  r |= dalloc(&e->ref, (size_t)B * m);
  r |= dalloc(&e->front, Bn * m);
  r |= dalloc(&e->mask, Bn);
  r |= dalloc(&e->P, (size_t)B);
  r |= dalloc(&e->K, (size_t)B);
  r |= dalloc(&e->lower, (size_t)B * cap * m);
  r |= dalloc(&e->upper, (size_t)B * cap * m);
  r |= dalloc(&e->Xc, BN * d);
  if (mode != BOUTE_ACQ_EHVI2D) r |= dalloc(&e->eps, BN * m * S);
  if (mode == BOUTE_ACQ_NEHVI) {
    const size_t zc = (size_t)B * m * S * n;
    r |= dalloc(&e->zin, zc);
    r |= dalloc(&e->Yin, zc);
    r |= dalloc(&e->shift, BN * m * S);
    r |= dalloc(&e->strips, (size_t)B * S * (n + 1) * 4);
    r |= dalloc(&e->counts, (size_t)B * S);
    if (r == BOUTE_OK) r = boute_gp_set_insample(e->gp, S);
    if (r == BOUTE_OK) r = draw_insample_normals(e, nullptr);  // seed 0 until set_normals
  }
  r |= dalloc(&e->mean, BN * m);
  r |= dalloc(&e->var, BN * m);
  r |= dalloc(&e->acq, BN);
  r |= dalloc(&e->idx, (size_t)B * k);
  r |= dalloc(&e->val, (size_t)B * k);
  r |= dalloc((unsigned char **)&e->scratch, topk_scratch_bytes(B, N, k));
  // the top-k counters in the scratch start at zero; every step leaves them zero
  if (r == BOUTE_OK && cudaMemset(e->scratch, 0, topk_scratch_bytes(B, N, k)) != cudaSuccess) {
    cudaGetLastError();
    r = BOUTE_ERR_CUDA;
  }
  e->fuse_sel = engine_fuses_selection(e);
  if (r == BOUTE_OK && e->fuse_sel) {
    const size_t bytes = e->sel_bytes = mchvi2_select_scratch_bytes(B, N, 2 * n + 2);
    r |= dalloc(&e->sel, bytes);
    if (r == BOUTE_OK && cudaMemset(e->sel, 0, bytes) != cudaSuccess) {
      cudaGetLastError();
      r = BOUTE_ERR_CUDA;
    }
  }
  if (r == BOUTE_OK && kstar_floats(&e->gp->g, N) * sizeof(float) <= kKstarMaxBytes)
    r |= dalloc(&e->kst, kstar_floats(&e->gp->g, N));
  if (r == BOUTE_OK &&
      (cudaStreamCreateWithFlags(&e->side, cudaStreamNonBlocking) != cudaSuccess ||
       cudaStreamCreateWithFlags(&e->side2, cudaStreamNonBlocking) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->ev_setup, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->join2, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->join, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->ev_in, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->ev_xc, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->ev_xc1, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->in_free[0], cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->in_free[1], cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->ev_small[0], cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&e->ev_small[1], cudaEventDisableTiming) != cudaSuccess)) {
    cudaGetLastError();
    r = BOUTE_ERR_CUDA;
  }
  for (int i = 0; r == BOUTE_OK && i < kCopyStreams; ++i)
    if (cudaStreamCreateWithFlags(&e->cpy[i], cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&e->ev_eps[i], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&e->ev_eps1[i], cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      r = BOUTE_ERR_CUDA;
    }
  if (r != BOUTE_OK) {
    boute_engine_free(e);
    return BOUTE_ERR_OOM;
  }
  *out = e;
  return BOUTE_OK;
}

static int engine_run(boute_engine *e, const double *X, const double *Y, const double *ls,
                      const double *s2, const double *noise, const double *ref, const float *Xc,
                      const float *eps, long long *idx, float *val, cudaStream_t s,
                      int host) {
  const unsigned long long l0 = launch_count();
  int r;
  const int B = e->B, n = e->n, m = e->m;
  const int mc = e->mode != BOUTE_ACQ_EHVI2D, nehvi = e->mode == BOUTE_ACQ_NEHVI;
  // stage boundaries: event-record nodes when captured, plain records when eager
  cudaStreamCaptureStatus run_cap = cudaStreamCaptureStatusNone;
  if (e->timing && s && cudaStreamIsCapturing(s, &run_cap) != cudaSuccess)
    return last_launch_status();
  // live timing (2): the normal schedule, events on the step's stream only
  const int serial = e->timing == 1, live = e->timing == 2;
  auto mark = [&](int stage) {
    if (!e->timing) return;
    if (run_cap == cudaStreamCaptureStatusActive)
      cudaEventRecordWithFlags(e->ev[stage], s, cudaEventRecordExternal);
    else
      cudaEventRecord(e->ev[stage], s);
  };
  auto front = [&](cudaStream_t fs) {
    return launch_front_fused(Y, B, n, m, ref, e->Ys, e->mask, e->front, e->P, e->lower,
                              e->upper, e->K, mc, fs);
  };
  mark(ST_FIT);
  // waits on the host-input copies: an external-event node when captured
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (host && cudaStreamIsCapturing(s, &cap) != cudaSuccess) return last_launch_status();
  const unsigned wait_flags =
      cap == cudaStreamCaptureStatusActive ? cudaEventWaitExternal : cudaEventWaitDefault;
  // host inputs: the copy events of input set host - 1
  const cudaEvent_t ev_xc = host == 2 ? e->ev_xc1 : e->ev_xc;
  const cudaEvent_t *ev_eps = host == 2 ? e->ev_eps1 : e->ev_eps;
  if (host && cudaStreamWaitEvent(s, e->ev_small[host - 1], wait_flags) != cudaSuccess)
    return last_launch_status();
  // outcome transforms: one elementwise pass first (the kernels after it see
  // transformed outcomes; without transforms the step does not have it)
  if (e->tcodes) {
    if ((r = launch_outcome_transform(Y, (long long)B * n * m, m, e->tcodes, e->Yt, s))) return r;
    Y = e->Yt;
  }
  // K* beside the fit (not in serialised timing, where the posterior builds it)
  const float *kst = serial ? nullptr : e->kst;
  // The graph has one root, the fit's set-up: the front stage (which needs
  // the raw outcomes only) and K* (which needs the set-up's side input) fork
  // after it and run beside the fit (one root launches sooner than two).
  if ((r = launch_fit_raw(&e->gp->g, X, Y, ls, s2, noise, s, serial ? nullptr : e->ev_setup)))
    return r;
  if (!serial) {
    if (cudaStreamWaitEvent(e->side, e->ev_setup, 0) != cudaSuccess) return last_launch_status();
    if ((r = front(e->side))) return r;
    if (cudaEventRecord(e->join, e->side) != cudaSuccess) return last_launch_status();
  }
  if (kst) {
    if (cudaStreamWaitEvent(e->side2, e->ev_setup, 0) != cudaSuccess ||
        (host && cudaStreamWaitEvent(e->side2, ev_xc, wait_flags) != cudaSuccess))
      return last_launch_status();
    if ((r = launch_kstar(&e->gp->g, Xc, e->N, e->kst, e->side2))) return r;
    if (cudaEventRecord(e->join2, e->side2) != cudaSuccess) return last_launch_status();
  }
  if (serial) {
    mark(ST_FRONT);
    if ((r = front(s))) return r;
    mark(ST_POSTERIOR);
  }
  if (nehvi) {  // the in-sample draws need the front stage's standardised outcomes
    if (!serial && cudaStreamWaitEvent(s, e->join, 0) != cudaSuccess) return last_launch_status();
    if ((r = launch_insample(&e->gp->g, e->Ys, s2, noise, e->zin, e->Yin, s))) return r;
  }
  if (host && cudaStreamWaitEvent(s, ev_xc, wait_flags) != cudaSuccess)
    return last_launch_status();
  if (kst && cudaStreamWaitEvent(s, e->join2, 0) != cudaSuccess) return last_launch_status();
  if (live) mark(ST_POSTERIOR);  // the posterior starts here (the front ran beside the fit)
  if ((r = nehvi ? launch_posterior_joint(&e->gp->g, Xc, e->N, e->mean, e->var, e->shift, s, kst)
                 : launch_posterior(&e->gp->g, Xc, e->N, e->mean, e->var, s, kst)))
    return r;
  if (live) mark(ST_ACQ);
  if (!serial && cudaStreamWaitEvent(s, e->join, 0) != cudaSuccess)  // join
    return last_launch_status();
  if (host && mc && eps != e->gen_eps)  // (the engine's own normals are resident)
    for (int i = 0; i < kCopyStreams; ++i)
      if (cudaStreamWaitEvent(s, ev_eps[i], wait_flags) != cudaSuccess)
        return last_launch_status();
  if (!live) mark(ST_ACQ);
  const double *cons = e->has_cons ? e->cons : nullptr;
  if (e->fuse_sel && !serial) {
    if ((r = launch_mchvi2_select(e->mean, e->var, B, e->N, e->lower, e->upper, e->K, 2 * n + 2,
                                  eps, e->S, 2ll * e->S, cons, e->acq, e->k, e->sel, idx, val,
                                  s)))
      return r;
  } else if (!mc) {
    if ((r = launch_ehvi(e->mean, e->var, B, e->N, e->front, e->P, n, ref, cons, e->acq, s)))
      return r;
  } else if (nehvi) {  // each draw's front, then the draws' improvements over them
    if ((r = launch_insample_fronts(e->Yin, B, n, e->S, ref, cons, e->strips, e->counts, s)) ||
        (r = launch_nehvi2(e->mean, e->var, e->shift, B, e->N, e->S, eps, 2ll * e->S, e->strips,
                           e->counts, n, cons, e->acq, s)))
      return r;
  } else {
    if ((r = launch_mchvi(e->mean, e->var, B, e->N, m, e->lower, e->upper, e->K, 2 * n + 2, eps,
                          e->S, (long long)m * e->S, cons, e->acq, s)))
      return r;
  }
  if (!e->fuse_sel || serial) {
    mark(ST_TOPK);
    if ((r = launch_topk(e->acq, B, e->N, e->k, idx, val, e->scratch, s, true))) return r;
  }
  mark(ST_COUNT);
  e->launches = (int)(launch_count() - l0);
  return BOUTE_OK;
}

static int engine_args_ok(const boute_engine *e, const void *X, const void *Y, const void *ls,
                          const void *s2, const void *noise, const void *ref, const void *Xc,
                          const void *eps, const void *idx, const void *val) {
  if (!e || !X || !Y || !ls || !s2 || !noise || !ref || !Xc || !idx || !val) return 0;
  if (e->mode != BOUTE_ACQ_EHVI2D && !eps && !e->gen_eps) return 0;
  return 1;
}

// Runs the step, through a cached CUDA graph when the stream can be captured.
static int engine_launch(boute_engine *e, const double *X, const double *Y, const double *ls,
                         const double *s2, const double *noise, const double *ref,
                         const float *Xc, const float *eps, long long *idx, float *val,
                         cudaStream_t s, int host = 0) {
  const void *key[12] = {X,   Y,   ls,  s2,  noise,           ref,
                         Xc,  eps, idx, val, (const void *)s, (const void *)(uintptr_t)host};
  if (!s || e->graphs_off)  // the legacy default stream cannot be captured
    return engine_run(e, X, Y, ls, s2, noise, ref, Xc, eps, idx, val, s, host);
  for (auto &g : e->graphs) {
    if (g.exec && std::memcmp(g.key, key, sizeof(key)) == 0) {
      if (cudaGraphLaunch(g.exec, s) != cudaSuccess) return last_launch_status();
      count_launch(g.launches);
      e->launches = g.launches;
      return BOUTE_OK;
    }
  }
  auto &g = e->graphs[e->graph_next];
  e->graph_next = (e->graph_next + 1) % 3;
  if (g.exec) {
    cudaGraphExecDestroy(g.exec);
    g.exec = nullptr;
  }
  if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    cudaGetLastError();
    return engine_run(e, X, Y, ls, s2, noise, ref, Xc, eps, idx, val, s, host);
  }
  const unsigned long long l0 = launch_count();
  const int r = engine_run(e, X, Y, ls, s2, noise, ref, Xc, eps, idx, val, s, host);
  cudaGraph_t graph = nullptr;
  const cudaError_t ce = cudaStreamEndCapture(s, &graph);
  const int captured = (int)(launch_count() - l0);
  g_launches_adjust(captured);  // the capture itself ran nothing
  if (r != BOUTE_OK || ce != cudaSuccess || !graph) {
    if (graph) cudaGraphDestroy(graph);
    cudaGetLastError();
    return r != BOUTE_OK ? r : BOUTE_ERR_CUDA;
  }
  cudaGraphExec_t exec = nullptr;
  const cudaError_t ie = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (ie != cudaSuccess) {
    cudaGetLastError();
    return BOUTE_ERR_CUDA;
  }
  std::memcpy(g.key, key, sizeof(key));
  g.exec = exec;
  g.launches = captured;
  if (cudaGraphLaunch(exec, s) != cudaSuccess) return last_launch_status();
  count_launch(captured);
  e->launches = captured;
  return BOUTE_OK;
}

int boute_engine_step_async(boute_engine *e, const double *X, const double *Y,
                            const double *lengthscale, const double *outputscale,
                            const double *noise, const double *ref, const float *Xc,
                            const float *eps, long long *idx, float *val, void *stream) {
  BOUTE_TRACE();
  if (!engine_args_ok(e, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx, val))
    return BOUTE_ERR_INVALID_ARG;
  if (!eps) eps = e->gen_eps;  // the engine's own normals (Monte-Carlo steps)
  return engine_launch(e, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx, val,
                       (cudaStream_t)stream);
}

// After a failed step the cross-block counters of the kernels that select as
// blocks finish may be left part-way: set them back to zero.
static void engine_reset_counters(boute_engine *e) {
  cudaDeviceSynchronize();
  cudaGetLastError();
  if (e->sel) cudaMemset(e->sel, 0, e->sel_bytes);
  cudaMemset(e->scratch, 0, topk_scratch_bytes(e->B, e->N, e->k));
  cudaGetLastError();
}

int boute_engine_step(boute_engine *e, const double *X, const double *Y,
                      const double *lengthscale, const double *outputscale, const double *noise,
                      const double *ref, const float *Xc, const float *eps, long long *idx,
                      float *val, void *stream) {
  BOUTE_TRACE();
  int r = boute_engine_step_async(e, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx,
                                  val, stream);
  if (!r) r = boute_gp_status(e->gp, stream);
  if (r && e) engine_reset_counters(e);
  return r;
}

// Copies a host-input step's inputs into device input set `set` and runs the
// step on `s`, its results copied back into idx / val (host); nothing waits.
// The inputs go on the two copy streams, after the last step that read this
// set (in_free), so that they overlap the previous step's computation: the
// small ones first, then the candidates, then the base normals in halves;
// the step waits for each only where it needs it (fit, posterior,
// acquisition).
static int engine_host_step(boute_engine *e, int set, const double *X, const double *Y,
                            const double *lengthscale, const double *outputscale,
                            const double *noise, const double *ref, const float *Xc,
                            const float *eps, long long *idx, float *val, cudaStream_t s) {
  const size_t B = e->B, n = e->n, d = e->d, m = e->m, N = e->N, S = e->S, k = e->k;
  double *dX = set ? e->X1 : e->X, *dY = set ? e->Y1 : e->Y, *dls = set ? e->ls1 : e->ls;
  double *ds2 = set ? e->s21 : e->s2, *dnz = set ? e->noise1 : e->noise;
  double *dref = set ? e->ref1 : e->ref;
  float *dXc = set ? e->Xc1 : e->Xc, *deps = set ? e->eps1 : e->eps;
  const cudaEvent_t ev_xc = set ? e->ev_xc1 : e->ev_xc;
  const cudaEvent_t *ev_eps = set ? e->ev_eps1 : e->ev_eps;
  for (cudaStream_t c : e->cpy) cudaStreamWaitEvent(c, e->in_free[set], 0);
  // the small inputs first, so that the step's fit never waits behind the
  // previous copies of the normals on the copy engine
  cudaStream_t c0 = e->cpy[0];
  cudaMemcpyAsync(dX, X, B * n * d * sizeof(double), cudaMemcpyHostToDevice, c0);
  cudaMemcpyAsync(dY, Y, B * n * m * sizeof(double), cudaMemcpyHostToDevice, c0);
  cudaMemcpyAsync(dls, lengthscale, B * m * d * sizeof(double), cudaMemcpyHostToDevice, c0);
  cudaMemcpyAsync(ds2, outputscale, B * m * sizeof(double), cudaMemcpyHostToDevice, c0);
  cudaMemcpyAsync(dnz, noise, B * m * sizeof(double), cudaMemcpyHostToDevice, c0);
  cudaMemcpyAsync(dref, ref, B * m * sizeof(double), cudaMemcpyHostToDevice, c0);
  cudaEventRecord(e->ev_small[set], c0);
  cudaMemcpyAsync(dXc, Xc, B * N * d * sizeof(float), cudaMemcpyHostToDevice, c0);
  cudaEventRecord(ev_xc, e->cpy[0]);
  const size_t eps_n = e->mode != BOUTE_ACQ_EHVI2D && eps ? B * N * m * S : 0;
  for (int i = 0; eps && i < kCopyStreams; ++i) {  // the normals in equal parts, one per stream
    const size_t off = eps_n * i / kCopyStreams, cnt = eps_n * (i + 1) / kCopyStreams - off;
    if (cnt)
      cudaMemcpyAsync(deps + off, eps + off, cnt * sizeof(float), cudaMemcpyHostToDevice,
                      e->cpy[i]);
    cudaEventRecord(ev_eps[i], e->cpy[i]);
  }
  if (!eps) deps = e->gen_eps;  // null: the engine's own normals
  if (int r = last_launch_status()) return r;
  int r = engine_launch(e, dX, dY, dls, ds2, dnz, dref, dXc, deps, e->idx, e->val, s, 1 + set);
  if (r) return r;
  cudaEventRecord(e->in_free[set], s);  // this step has read set `set`
  cudaMemcpyAsync(idx, e->idx, B * k * sizeof(long long), cudaMemcpyDeviceToHost, s);
  cudaMemcpyAsync(val, e->val, B * k * sizeof(float), cudaMemcpyDeviceToHost, s);
  return last_launch_status();
}

int boute_engine_step_host(boute_engine *e, const double *X, const double *Y,
                           const double *lengthscale, const double *outputscale,
                           const double *noise, const double *ref, const float *Xc,
                           const float *eps, long long *idx, float *val, void *stream) {
  BOUTE_TRACE();
  if (!engine_args_ok(e, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx, val))
    return BOUTE_ERR_INVALID_ARG;
  int r = engine_host_step(e, 0, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx, val,
                           (cudaStream_t)stream);
  if (!r) r = boute_gp_status(e->gp, stream);
  if (r) engine_reset_counters(e);
  return r;
}

int boute_engine_step_host_async(boute_engine *e, const double *X, const double *Y,
                                 const double *lengthscale, const double *outputscale,
                                 const double *noise, const double *ref, const float *Xc,
                                 const float *eps, long long *idx, float *val, void *stream) {
  BOUTE_TRACE();
  if (!engine_args_ok(e, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx, val))
    return BOUTE_ERR_INVALID_ARG;
  if (!e->X1) {  // the second input set, on first use
    const size_t Bn = (size_t)e->B * e->ncap, BN = (size_t)e->B * e->N, Bm = (size_t)e->B * e->m;
    int r = dalloc(&e->X1, Bn * e->d) | dalloc(&e->Y1, Bn * e->m) |
            dalloc(&e->ls1, Bm * e->d) | dalloc(&e->s21, Bm) | dalloc(&e->noise1, Bm) |
            dalloc(&e->ref1, Bm) | dalloc(&e->Xc1, BN * e->d);
    if (e->mode != BOUTE_ACQ_EHVI2D) r |= dalloc(&e->eps1, BN * e->m * e->S);
    if (r) return BOUTE_ERR_OOM;
  }
  const int set = e->host_set;
  e->host_set ^= 1;
  return engine_host_step(e, set, X, Y, lengthscale, outputscale, noise, ref, Xc, eps, idx, val,
                          (cudaStream_t)stream);
}

int boute_engine_sync(boute_engine *e, void *stream) {
  BOUTE_TRACE();
  if (!e) return BOUTE_ERR_INVALID_ARG;
  const int r = boute_gp_status(e->gp, stream);
  if (r) engine_reset_counters(e);
  return r;
}

int boute_engine_scores(const boute_engine *e, float *acq, float *mean, float *var,
                        void *stream) {
  BOUTE_TRACE();
  if (!e) return BOUTE_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  const size_t BN = (size_t)e->B * e->N;
  if (acq) cudaMemcpyAsync(acq, e->acq, BN * sizeof(float), cudaMemcpyDeviceToDevice, s);
  if (mean) cudaMemcpyAsync(mean, e->mean, BN * e->m * sizeof(float), cudaMemcpyDeviceToDevice, s);
  if (var) cudaMemcpyAsync(var, e->var, BN * e->m * sizeof(float), cudaMemcpyDeviceToDevice, s);
  return last_launch_status();
}

int boute_engine_set_timing(boute_engine *e, int on) {
  BOUTE_TRACE();
  if (!e) return BOUTE_ERR_INVALID_ARG;
  if (on < 0 || on > 2) return BOUTE_ERR_INVALID_ARG;
  if (on == e->timing) return BOUTE_OK;
  if (on && !e->ev[0])
    for (int i = 0; i <= ST_COUNT; ++i)
      if (cudaEventCreate(&e->ev[i]) != cudaSuccess) return last_launch_status();
  e->timing = on;
  for (auto &g : e->graphs)  // recapture: event nodes in or out, front stage placement
    if (g.exec) {
      cudaGraphExecDestroy(g.exec);
      g.exec = nullptr;
    }
  return BOUTE_OK;
}

int boute_engine_stage_times(boute_engine *e, float *ms, int count) {
  BOUTE_TRACE();
  if (!e || !ms || count < ST_COUNT || !e->ev[0]) return BOUTE_ERR_INVALID_ARG;
  if (cudaEventSynchronize(e->ev[ST_COUNT]) != cudaSuccess) return last_launch_status();
  if (e->timing == 2) {
    // live: no front boundary (it ran beside the fit); with the selection
    // inside the acquisition kernel no top-k boundary either
    const bool sel = e->fuse_sel != 0;
    const int acq_end = sel ? ST_COUNT : ST_TOPK;
    ms[ST_FRONT] = 0.f;
    if (sel) ms[ST_TOPK] = 0.f;
    if (cudaEventElapsedTime(&ms[ST_FIT], e->ev[ST_FIT], e->ev[ST_POSTERIOR]) != cudaSuccess ||
        cudaEventElapsedTime(&ms[ST_POSTERIOR], e->ev[ST_POSTERIOR], e->ev[ST_ACQ]) !=
            cudaSuccess ||
        cudaEventElapsedTime(&ms[ST_ACQ], e->ev[ST_ACQ], e->ev[acq_end]) != cudaSuccess ||
        (!sel &&
         cudaEventElapsedTime(&ms[ST_TOPK], e->ev[ST_TOPK], e->ev[ST_COUNT]) != cudaSuccess))
      return last_launch_status();
    return BOUTE_OK;
  }
  for (int i = 0; i < ST_COUNT; ++i)
    if (cudaEventElapsedTime(&ms[i], e->ev[i], e->ev[i + 1]) != cudaSuccess)
      return last_launch_status();
  return BOUTE_OK;
}

int boute_engine_launches_per_step(const boute_engine *e) { return e ? e->launches : 0; }

// the cached step graphs hold kernel arguments and kernel choices: drop them
static void engine_drop_graphs(boute_engine *e) {
  for (auto &g : e->graphs)
    if (g.exec) {
      cudaGraphExecDestroy(g.exec);
      g.exec = nullptr;
    }
}

// Re-plan the handle for n <= ncap observations: the posterior's operand
// layout (plan), its K* cache share, and zero padding in the operand images
// and side inputs (their strides change with n).
static int gp_set_n(Gp &g, int n) {
  if (n < 1 || n > g.ncap) return BOUTE_ERR_INVALID_ARG;
  if (n == g.n) return BOUTE_OK;
  const size_t BM = (size_t)g.B * g.m;
  const int S_in = g.plan.S_in;
  const PostPlan cap = make_post_plan(g.ncap, S_in);
  g.n = n;
  g.plan = make_post_plan(n, S_in);
  const int want = kstar_cache_chunks(g.plan);
  g.kcache_chunks = want <= g.kcache_cap ? want : 0;  // else K* is rebuilt, not cached
  if (cudaMemset(g.bop, 0, BM * (size_t)cap.image_halves * sizeof(uint16_t)) != cudaSuccess ||
      cudaMemset(g.xt, 0, BM * (size_t)cap.nxt * xt_chunk_floats(g.DP) * sizeof(float)) !=
          cudaSuccess) {
    cudaGetLastError();
    return BOUTE_ERR_CUDA;
  }
  return BOUTE_OK;
}

int boute_engine_optimize(boute_engine *e, const float *eps, int S, const float *X0, int P,
                          const float *xlo, const float *xhi, int steps, float lr, float *X,
                          float *acq, float *grad, void *stream) {
  BOUTE_TRACE();
  if (!e) return BOUTE_ERR_INVALID_ARG;
  if (e->mode != BOUTE_ACQ_MC_HVI || e->m != 2) return BOUTE_ERR_UNSUPPORTED;
  return boute_acq_optimize(e->gp, e->lower, e->upper, e->K, 2 * e->n + 2, eps, S, X0, P, xlo,
                            xhi, steps, lr, X, acq, grad, stream);
}

int boute_engine_set_n(boute_engine *e, int n) {
  BOUTE_TRACE();
  if (!e || n < 1 || n > e->ncap) return BOUTE_ERR_INVALID_ARG;
  if (n == e->n) return BOUTE_OK;
  if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  if (int r = gp_set_n(e->gp->g, n)) return r;
  e->n = n;
  engine_drop_graphs(e);  // the graphs hold n and the plan in their arguments
  if (e->mode == BOUTE_ACQ_NEHVI) {  // the in-sample normals in the layout of n
    if (int r = draw_insample_normals(e, nullptr)) return r;
    if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  }
  // the in-kernel selection's scratch grows as the boxes shrink (more
  // resident blocks): keep it when it is large enough, else take a new one
  e->fuse_sel = engine_fuses_selection(e);
  if (e->fuse_sel) {
    const size_t bytes = mchvi2_select_scratch_bytes(e->B, e->N, 2 * n + 2);
    if (bytes > e->sel_bytes) {
      cudaFree(e->sel);
      e->sel = nullptr;
      e->sel_bytes = 0;
      if (dalloc(&e->sel, bytes) != BOUTE_OK) {
        e->fuse_sel = false;
        return BOUTE_ERR_OOM;
      }
      e->sel_bytes = bytes;
      if (cudaMemset(e->sel, 0, bytes) != cudaSuccess) {
        cudaGetLastError();
        return BOUTE_ERR_CUDA;
      }
    }
  }
  return BOUTE_OK;
}

int boute_engine_set_kernel(boute_engine *e, int d_tau, const double *params) {
  BOUTE_TRACE();
  if (!e) return BOUTE_ERR_INVALID_ARG;
  const int r = boute_gp_set_kernel(e->gp, d_tau, params);
  engine_drop_graphs(e);  // the step's kernel choices change
  return r;
}

int boute_acq_optimize(const boute_gp *gp, const float *lower, const float *upper, const int *K,
                       int box_cap, const float *eps, int S, const float *X0, int P,
                       const float *xlo, const float *xhi, int steps, float lr, float *X,
                       float *acq, float *grad, void *stream) {
  BOUTE_TRACE();
  if (!gp || !lower || !upper || !K || !eps || !X0 || !xlo || !xhi || !X || !acq || box_cap < 1 ||
      S < 1 || P < 1 || steps < 0 || !(lr > 0.f) || P > 65535)
    return BOUTE_ERR_INVALID_ARG;
  return launch_acq_optimize(&gp->g, lower, upper, K, box_cap, eps, S, X0, P, xlo, xhi, steps, lr,
                             X, acq, grad, (cudaStream_t)stream);
}

int boute_bounds_report(long long *rec) {
  BOUTE_TRACE();
  if (!rec) return BOUTE_ERR_INVALID_ARG;
#ifndef BOUTE_DEBUG_BOUNDS
  rec[0] = rec[1] = rec[2] = rec[3] = 0;
  return BOUTE_ERR_UNSUPPORTED;
#else
  if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  int (*readers[])(long long *) = {bounds_read_posterior, bounds_read_insample, bounds_read_acq,
                                   bounds_read_front,     bounds_read_fit,      bounds_read_topk};
  int found = 0;
  rec[0] = rec[1] = rec[2] = rec[3] = 0;
  for (int u = 0; u < (int)(sizeof(readers) / sizeof(readers[0])); ++u) {
    long long r[4];
    if (readers[u](r) != 0) return BOUTE_ERR_CUDA;
    if (r[0] && !found) {  // the first unit with a record; every record is cleared
      rec[0] = u + 1;
      rec[1] = r[1];
      rec[2] = r[2];
      rec[3] = r[3];
      found = 1;
    }
  }
  return found;
#endif
}

int boute_selftest_wait(int complete, unsigned long long limit_ns, void *stream) {
  BOUTE_TRACE();
  if (limit_ns > BOUTE_WAIT_NS) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  cudaStream_t s = (cudaStream_t)stream;
  int *status = nullptr;
  if (dalloc(&status, 1) != BOUTE_OK) return BOUTE_ERR_OOM;
  int r = cudaMemsetAsync(status, 0, sizeof(int), s) == cudaSuccess ? BOUTE_OK : BOUTE_ERR_CUDA;
  if (!r) r = launch_wait_selftest(complete, limit_ns, status, s);
  int st = BOUTE_OK;
  if (!r && (cudaStreamSynchronize(s) != cudaSuccess ||
             cudaMemcpy(&st, status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess))
    r = last_launch_status();
  cudaFree(status);
  return r ? r : st;
}

int boute_base_normals(unsigned long long seed, int B, long long N, int m, int S, float *eps,
                       void *stream) {
  BOUTE_TRACE();
  if (B < 1 || N < 0 || m < 1 || S < 1 || (N > 0 && !eps)) return BOUTE_ERR_INVALID_ARG;
  if (int r = device_ok()) return r;
  return launch_base_normals(seed, B, N, m, S, eps, (cudaStream_t)stream);
}

int boute_engine_set_normals(boute_engine *e, unsigned long long seed) {
  BOUTE_TRACE();
  if (!e || e->mode == BOUTE_ACQ_EHVI2D) return BOUTE_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  const size_t count = (size_t)e->B * e->N * e->m * e->S;
  if (!e->gen_eps && dalloc(&e->gen_eps, count) != BOUTE_OK) return BOUTE_ERR_OOM;
  int r = launch_base_normals(seed, e->B, e->N, e->m, e->S, e->gen_eps, nullptr);
  if (!r && e->mode == BOUTE_ACQ_NEHVI) {
    e->zseed = seed;
    r = draw_insample_normals(e, nullptr);
  }
  if (!r && cudaDeviceSynchronize() != cudaSuccess) r = last_launch_status();
  return r;
}

int boute_engine_set_outcome_transforms(boute_engine *e, const int *codes) {
  BOUTE_TRACE();
  int packed = 0;
  if (!e || !pack_codes(codes, e->m, &packed)) return BOUTE_ERR_INVALID_ARG;
  if (packed != e->tcodes) {
    if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
    if (packed && !e->Yt && dalloc(&e->Yt, (size_t)e->B * e->ncap * e->m) != BOUTE_OK)
      return BOUTE_ERR_OOM;
    e->tcodes = packed;
    engine_drop_graphs(e);
  }
  return BOUTE_OK;
}

int boute_engine_set_constraints(boute_engine *e, const double *cons) {
  BOUTE_TRACE();
  if (!e) return BOUTE_ERR_INVALID_ARG;
  const size_t count = (size_t)e->B * e->m;
  for (size_t i = 0; cons && i < count; ++i)
    if (cons[i] != cons[i]) return BOUTE_ERR_INVALID_ARG;  // NaN: no threshold
  // no step of this engine may be reading the thresholds while they change
  if (cudaDeviceSynchronize() != cudaSuccess) return last_launch_status();
  if (cons) {
    if (!e->cons && dalloc(&e->cons, count) != BOUTE_OK) return BOUTE_ERR_OOM;
    if (cudaMemcpy(e->cons, cons, count * sizeof(double), cudaMemcpyHostToDevice) != cudaSuccess)
      return last_launch_status();
  }
  const int on = cons != nullptr;
  if (on != e->has_cons) {  // the step's acquisition kernel changes: recapture
    e->has_cons = on;
    engine_drop_graphs(e);
  }
  return BOUTE_OK;
}

}  // extern "C"
