// Host-side declarations shared by the translation units of libboute.
#pragma once

#include <cuda_runtime.h>

#include "bounds.cuh"
#include "common.cuh"

#include <nvtx3/nvToolsExt.h>

namespace boute {

// The boute_gp handle: fp64 factors plus the prepacked tensor-core operands.
struct Gp {
  int B, n, d, m, DP;  // DP = d rounded up to a multiple of 4 (register tile)
  PostPlan plan;
  float *Kh, *Kl;  // B*m x n x n: kernel matrix (lower) as an fp32 pair hi + lo
  float *Aws;      // B*m x np x (np+1): factorisation workspace (large n; np = npad)
  float *Wws;      // B*m x np x (np+1): L^-1 (lower, row stride np+1)
  uint16_t *bop;  // B*m x plan.image_halves: L^-1 as fp16 hi/lo operand images
  // the posterior's cache of K* chunks that later groups of output blocks
  // need again (n > 512): kcache_chunks fp16 A-stage images per SM
  uint16_t *kcache;
  int kcache_chunks, kcache_sms;
  // capacity: the buffers above are sized for ncap observations; n <= ncap
  // (an engine re-plans its handle for each n of a growing data set)
  int ncap, kcache_cap;
  float *xt;      // B*m x nxt x xt_chunk_floats(DP): X/lengthscale hi/lo, alpha
  float *s2f;     // B*m: outputscale
  int *status;    // device status word (first error wins)
  int *fbad;      // B*m: a non-positive pivot in the blocked factorisation (n > 160)
  float *tpart;   // the blocked factorisation's partial sums of T_pJ (fit_tpart_floats)
  float *fvec;    // the blocked path's alpha vectors (fit_fvec_floats)
  // the FP64 tier (prec = BOUTE_PREC_FP64): W = L^-1 (B*m x n x n), alpha
  // (B*m x n), X / lengthscale (B*m x n x d), lengthscales (B*m x d) and
  // outputscales (B*m) of the last fit, all fp64
  int prec;
  double *W64, *a64, *xs64, *ls64, *s2_64;
  // the composite kernel (kern = 1): routing features [0, dtau) and per
  // problem-objective [s2_c, s2_x, beta, s_0 .. s_{d-1}] (B*m x (3 + d))
  int kern, dtau;
  double *kpar;
  // in-sample draws of the noisy acquisition (plan.S_in > 0, n <= kInsMaxN):
  // G^T = (H Z)^T, S_in x n per problem-objective, before it is packed, and
  // the preparation's workspace (F, H^T, mu_n, max |G|: insample_ws_floats)
  float *gws, *iws;
};

// An NVTX range over one call of the C-ABI (visible in a profiler's timeline;
// a few nanoseconds when no tool is attached).
struct TraceRange {
  explicit TraceRange(const char *name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange &) = delete;
  TraceRange &operator=(const TraceRange &) = delete;
};
#define BOUTE_TRACE() ::boute::TraceRange boute_trace_range_(__func__)

// Every kernel of the step asks for the largest shared-memory carveout, so
// that consecutive kernels never make an SM switch its L1 / shared split.
template <class F>
inline void prefer_shared(F *kernel) {
  cudaFuncSetAttribute((const void *)kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                       (int)cudaSharedmemCarveoutMaxShared);
}

// Launch with programmatic stream serialization: the kernel may begin while
// the previous kernel on the stream finishes, and waits (pdl_wait) before
// reading its results.
template <class... KArgs, class... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

inline int num_sms() {
  int dev = 0, sms = 152;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms;
}

// floats of the blocked factorisation's partial-sum workspace for B*m = BM
// problem-objectives at padded size npad (0 when that size never takes it)
size_t fit_tpart_floats(int npad, int BM);
// floats of the blocked path's alpha vectors (0 likewise)
size_t fit_fvec_floats(int npad, int BM);

void count_launch(int k = 1);
unsigned long long launch_count();
int last_launch_status();  // BOUTE_OK or BOUTE_ERR_CUDA after a launch

// FP64 tier (n <= 128, Matern-5/2): the fit's fp64 factor and the posterior
int launch_fit64(Gp *gp, const double *X, const double *Ys, const double *ls, const double *s2,
                 const double *noise, cudaStream_t s);
int launch_posterior64(const Gp *gp, const float *Xc, long long N, double *mean, double *var,
                       cudaStream_t s);
constexpr int kFp64MaxN = 128;
// Noisy acquisition (Sec. 5.2): the in-sample preparation after a fit (the
// in-sample draws Yin, and H, G into the operand images; n <= kInsMaxN), the
// fronts of the draws and the acquisition over them (two objectives).
constexpr int kInsMaxN = 128, kInsMaxS = 1024;
constexpr double kInsJitter = 1e-8;  // times the outputscale
int launch_insample(Gp *gp, const double *Ys, const double *s2, const double *noise,
                    const float *z, float *Yin, cudaStream_t s);
size_t insample_smem_bytes(int n);
size_t insample_ws_floats(int n);  // per problem-objective
int launch_insample_fronts(const float *Yin, int B, int n, int S, const double *ref,
                           const double *cons, float *strips, int *counts, cudaStream_t s);
int launch_nehvi2(const float *mean, const float *cvar, const float *shift, int B, long long N,
                  int S, const float *eps, long long eps_stride, const float *strips,
                  const int *counts, int n, const double *cons, float *acq, cudaStream_t s);
// Projected Adam ascent on the 2-objective sample-average MC acquisition
// from P starting points per problem (acqopt.cu).
int launch_acq_optimize(const Gp *gp, const float *lower, const float *upper, const int *K,
                        int box_cap, const float *eps, int S, const float *X0, int P,
                        const float *xlo, const float *xhi, int steps, float lr, float *X,
                        float *acq, float *grad, cudaStream_t s);
// The posterior with the in-sample blocks: mean, the conditional variance
// (cvar) and the shifts (B x m x S_in x N); shift null: the plain posterior
// (W's blocks only) on a handle with in-sample draws.
int launch_posterior_joint(const Gp *gp, const float *Xc, long long N, float *mean, float *cvar,
                           float *shift, cudaStream_t s, const float *kst = nullptr);
// the library's device check (an sm_103a device is current)
int device_ok();
// bounds records of the debug build, per translation unit (bounds.cuh)
int bounds_read_posterior(long long *out);
int bounds_read_insample(long long *out);
int bounds_read_acq(long long *out);
int bounds_read_front(long long *out);
int bounds_read_fit(long long *out);
int bounds_read_topk(long long *out);
// codes: outcome transforms before standardising (objective_code)
int launch_standardize(const double *Y, int B, int n, int m, int codes, double *Ys,
                       cudaStream_t s);
int launch_fit(Gp *gp, const double *X, const double *Ys, const double *ls, const double *s2,
               const double *noise, cudaStream_t s);
// kst: K* precomputed by launch_kstar (the posterior then builds no K*), or null.
int launch_posterior(const Gp *gp, const float *Xc, long long N, float *mean, float *var,
                     cudaStream_t s, const float *kst = nullptr);
// Chunks of K* per CTA that the posterior caches across groups of output
// blocks (0 when every chunk is needed by one group only).
int kstar_cache_chunks(const PostPlan &plan);
// fp16 halves of one cached chunk (an A stage: 128 x 64 hi and lo)
constexpr size_t kKstarChunkHalves = 2 * BOUTE_TILE_M * BOUTE_ACHUNK;
// K* of all candidates, per (128-candidate tile, objective) and 64-point chunk
// as the fp16 hi and lo images of an A stage (128 x 64 each, scaled by the
// row's 2^e_r): kstar_floats(gp, N) 4-byte words. Reads the fit set-up's side
// input (not the fit's results) and the candidates.
size_t kstar_floats(const Gp *gp, long long N);
int launch_kstar(const Gp *gp, const float *Xc, long long N, float *kst, cudaStream_t s);
int launch_pareto(const double *Ys, int B, int n, int m, const double *ref, unsigned char *mask,
                  double *front, int *P, cudaStream_t s);
size_t front_smem_bytes(int n, int m);
int launch_front_fused(const double *Y, int B, int n, int m, const double *ref, double *Ys,
                       unsigned char *mask, double *front, int *P, float *lower, float *upper,
                       int *K, int want_boxes, cudaStream_t s);
// Yt = outcome transforms (objective_code) of Y, count values, m objectives
int launch_outcome_transform(const double *Y, long long count, int m, int codes, double *Yt,
                             cudaStream_t s);
// setup_done (optional) is recorded on s after the set-up kernel, before the fit.
int launch_fit_raw(Gp *gp, const double *X, const double *Y, const double *ls, const double *s2,
                   const double *noise, cudaStream_t s,
                   cudaEvent_t setup_done = nullptr);
int launch_boxes(const double *front, const int *P, int B, int n, int m, const double *ref,
                 float *lower, float *upper, int *K, cudaStream_t s);
// cons: per problem m thresholds on the minimised objectives (device), or null
int launch_ehvi(const float *mean, const float *var, int B, long long N, const double *front,
                const int *P, int n, const double *ref, const double *cons, float *acq,
                cudaStream_t s);
unsigned mchvi2_select_grid_x(int B, long long N, int box_cap);
size_t mchvi2_select_scratch_bytes(int B, long long N, int box_cap);
int launch_mchvi2_select(const float *mean, const float *var, int B, long long N,
                         const float *lower, const float *upper, const int *K, int box_cap,
                         const float *eps, int S, long long eps_stride, const double *cons,
                         float *acq, int k, void *sel, long long *idx, float *val,
                         cudaStream_t s);
int launch_mchvi(const float *mean, const float *var, int B, long long N, int m,
                 const float *lower, const float *upper, const int *K, int box_cap,
                 const float *eps, int S, long long eps_stride, const double *cons, float *acq,
                 cudaStream_t s);
// hyperparameter learning (learn.cu): B*m*R blocks, fp64; workspace from the
// stream-ordered pool when a block's does not fit in shared memory
// dtau, pref: the composite kernel's routing features and preference entries
// (B x m x (d - dtau)); pref null: the Matern-5/2 kernel
int launch_learn(const double *X, const double *Ys, int B, int n, int d, int m,
                 const double *theta0, int R, int iters, double lr, double *theta, double *mll,
                 double *grad, int dtau, const double *pref, cudaStream_t s);
// Monte-Carlo base normals from Philox4x64-10 and Box-Muller (B x N x m x S)
int launch_base_normals(unsigned long long seed, int B, long long N, int m, int S, float *eps,
                        cudaStream_t s);
// a bounded device-side wait that runs out unless `complete` (selftest.cu)
int launch_wait_selftest(int complete, unsigned long long limit_ns, int *status, cudaStream_t s);
size_t topk_scratch_bytes(int B, long long N, int k);
// counters_zeroed: the scratch's per-problem counters are known to be zero
// (an engine's scratch: zeroed at creation, and every call leaves them zero);
// otherwise the call clears them first.
int launch_topk(const float *acq, int B, long long N, int k, long long *idx, float *val,
                void *scratch, cudaStream_t s, bool counters_zeroed = false);

}  // namespace boute
