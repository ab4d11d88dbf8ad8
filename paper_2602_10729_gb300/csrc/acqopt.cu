// Optimising the acquisition over the decision space (Sec. 5.2 step (ii),
// "optimize it over the decision space"): projected Adam ascent on the
// sample-average Monte-Carlo hypervolume improvement of two objectives, from
// given starting points (for instance the best candidates of a pool).
//
// With fixed base normals eps_s the acquisition A(x) = (1/S) sum_s HVI(mu(x) +
// sd(x) eps_s) is a deterministic, piecewise smooth function of x. Its
// gradient runs through the GP posterior of each objective (Matern-5/2):
//   k*_j = s2 (1 + sqrt5 r + 5/3 r^2) e^(-sqrt5 r),
//   dk*_j/dx_k = -5/3 s2 (1 + sqrt5 r) e^(-sqrt5 r) (x_k - X_jk) / l_k^2,
//   mu = k*^T alpha,  var = s2 - |W k*|^2,  dvar/dx = -2 (W^T W k*)^T dk*/dx,
// and the strip sum HVI(y) = sum_k (b_k - max(a_k, y1))+ (u_k - y2)+, whose
// derivatives are -(u_k - y2)+ for the strip containing y1 and
// -sum_k (b_k - max(a_k, y1))+ [y2 < u_k].
//
// One CTA per (problem, starting point) runs all its steps: per step and
// objective the threads build k* and its gradient factors over the training
// points (the fit's side input: scaled coordinates hi + lo, alpha as a pair),
// form W k* (a warp per row) and W^T (W k*) (a thread per column) from the
// fit's W, reduce the mean, variance and their gradients, then score the S
// draws (a thread per draw) against the observed front's strips.
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace boute {

namespace {

constexpr int kOptThreads = 128, kOptWarps = kOptThreads / 32;
constexpr float kLn2f = 0.6931471805599453f;
constexpr float kLn2Sq3f = 0.16015100463940046f;  // (ln 2)^2 / 3
// 1 / (the side input's coordinate scale)^2
constexpr float kInvScale2 = (float)(1.0 / (kCoordScale52 * kCoordScale52));

struct OptArgs {
  const float *Wws, *xt;
  int npad, nxt, DP, n, d, m;
  const float *lower, *upper;  // the observed front's strips (box decomposition)
  const int *K;
  int box_cap;
  const float *eps;  // 2 x S, shared by every point
  int S;
  const float *X0, *xlo, *xhi;
  int P, steps;
  float lr;
  float *X, *acq, *grad;
};

// block-wide sum of v (every thread receives it)
__device__ __forceinline__ float block_sum(float v, float *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int w = 0; w < kOptWarps; ++w) s += red[w];
  return s;
}

__global__ void __launch_bounds__(kOptThreads) acqopt_kernel(const __grid_constant__ OptArgs a) {
  extern __shared__ __align__(16) float sm[];
  __shared__ float red[kOptWarps];
  __shared__ float xs[BOUTE_MAX_D], gx[BOUTE_MAX_D], m1[BOUTE_MAX_D], m2[BOUTE_MAX_D];
  __shared__ float mu_s[2], sd_s[2], dmu_s[2][BOUTE_MAX_D], dsd_s[2][BOUTE_MAX_D], coef[5];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.y, p = blockIdx.x;
  const int n = a.n, d = a.d, DP = a.DP, cf = xt_chunk_floats(DP);
  float *kv = sm, *cv = kv + n, *qv = cv + n, *wv = qv + n;  // k*, c_j, W k*, W^T W k*
  float *df = wv + n;                                        // n x d scaled differences / l
  pdl_wait();
  for (int k = tid; k < d; k += kOptThreads) {
    xs[k] = a.X0[((size_t)b * a.P + p) * d + k];
    m1[k] = m2[k] = 0.f;
  }
  __syncthreads();
  const int K = BOUTE_INB(a.K[b], a.box_cap + 1) ? a.K[b] : 0;
  const float *lo = a.lower + (size_t)b * a.box_cap * 2, *up = a.upper + (size_t)b * a.box_cap * 2;
  float val = 0.f;
  for (int it = 0; it <= a.steps; ++it) {
    // ---- the posterior of both objectives at x, and its gradient
    for (int t = 0; t < 2; ++t) {
      const int bt = b * a.m + t;
      const float *x0 = a.xt + (size_t)bt * a.nxt * cf;
      const float *par = x0 + xt_param_offset(DP);  // 1/l hi [DP], 1/l lo [DP], scalars
      const float s2 = par[2 * DP + kParS2];
      float amu = 0.f;
      for (int j = tid; j < n; j += kOptThreads) {
        const float *ch = x0 + (size_t)(j / BOUTE_KCHUNK) * cf;
        const int jj = j % BOUTE_KCHUNK;
        float r2 = 0.f;
        for (int k = 0; k < d; ++k) {
          const float xk = fmaf(xs[k], par[k], xs[k] * par[DP + k]);  // x_k / l_k
          const float dk = (xk - ch[k * BOUTE_KCHUNK + jj]) - ch[(DP + k) * BOUTE_KCHUNK + jj];
          df[(size_t)j * d + k] = dk * (par[k] + par[DP + k]) * kInvScale2;  // (x_k - X_jk) / l_k^2
          r2 = fmaf(dk, dk, r2);
        }
        // r2 = r'^2, the side input's scaled distance: sqrt5 r = ln2 r',
        // exp(-sqrt5 r) = 2^(-r'); df above carries the scale twice
        const float rs = sqrtf(r2), ex = exp2f(-rs);
        kv[j] = s2 * fmaf(kLn2Sq3f, r2, fmaf(kLn2f, rs, 1.f)) * ex;
        cv[j] = -5.f / 3.f * s2 * fmaf(kLn2f, rs, 1.f) * ex;
        const float *al = ch + xt_alpha_offset(DP) + jj;
        amu = fmaf(kv[j], al[0] + al[BOUTE_KCHUNK], amu);
      }
      const float mu = block_sum(amu, red);  // (its barriers publish kv, cv, df)
      // q = W k* (a warp per row), then w = W^T q (a thread per column)
      const float *W = a.Wws + (size_t)bt * a.npad * (a.npad + 1);
      for (int i = warp; i < n; i += kOptWarps) {
        float s = 0.f;
        for (int j = lane; j <= i; j += 32) s = fmaf(W[(size_t)i * (a.npad + 1) + j], kv[j], s);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) qv[i] = s;
      }
      __syncthreads();
      float aq = 0.f;
      for (int j = tid; j < n; j += kOptThreads) {
        float s = 0.f;
        for (int i = j; i < n; ++i) s = fmaf(W[(size_t)i * (a.npad + 1) + j], qv[i], s);
        wv[j] = s;
        aq = fmaf(qv[j], qv[j], aq);
      }
      const float var = fmaxf(s2 - block_sum(aq, red), 0.f);
      // d mu / dx_k = sum_j alpha_j c_j df_jk, d var / dx_k = -2 sum_j w_j c_j df_jk
      for (int k = warp; k < d; k += kOptWarps) {
        float gm = 0.f, gv = 0.f;
        for (int j = lane; j < n; j += 32) {
          const float *al = x0 + (size_t)(j / BOUTE_KCHUNK) * cf + xt_alpha_offset(DP) + j % 32;
          const float cd = cv[j] * df[(size_t)j * d + k];
          gm = fmaf(al[0] + al[BOUTE_KCHUNK], cd, gm);
          gv = fmaf(wv[j], cd, gv);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          gm += __shfl_xor_sync(0xffffffffu, gm, o);
          gv += __shfl_xor_sync(0xffffffffu, gv, o);
        }
        if (lane == 0) {
          const float sd = sqrtf(var);
          dmu_s[t][k] = gm;
          dsd_s[t][k] = sd > 0.f ? -gv / sd : 0.f;  // d sd = d var / (2 sd)
        }
      }
      if (tid == 0) {
        mu_s[t] = mu;
        sd_s[t] = sqrtf(var);
      }
      __syncthreads();
    }
    // ---- the draws against the front's strips: A, dA/dmu_t, dA/dsd_t
    float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
    for (int s = tid; s < a.S; s += kOptThreads) {
      const float e0 = a.eps[s], e1 = a.eps[a.S + s];
      const float y1 = fmaf(sd_s[0], e0, mu_s[0]), y2 = fmaf(sd_s[1], e1, mu_s[1]);
      float h = 0.f, g1 = 0.f, g2 = 0.f;
      for (int k = 0; k < K; ++k) {
        const float ak = lo[2 * k], bk = up[2 * k], uk = up[2 * k + 1];
        const float wdt = fmaxf(bk - fmaxf(ak, y1), 0.f), hgt = fmaxf(uk - y2, 0.f);
        h = fmaf(wdt, hgt, h);
        if (ak < y1 && y1 < bk) g1 -= hgt;
        if (y2 < uk) g2 -= wdt;
      }
      acc[0] += h;
      acc[1] += g1;
      acc[2] += g1 * e0;
      acc[3] += g2;
      acc[4] += g2 * e1;
    }
    for (int q = 0; q < 5; ++q) {
      const float v = block_sum(acc[q], red);
      if (tid == 0) coef[q] = v / (float)a.S;
    }
    __syncthreads();
    val = coef[0];
    for (int k = tid; k < d; k += kOptThreads)
      gx[k] = coef[1] * dmu_s[0][k] + coef[2] * dsd_s[0][k] + coef[3] * dmu_s[1][k] +
              coef[4] * dsd_s[1][k];
    __syncthreads();
    if (it == a.steps) break;  // the last pass only evaluates
    // ---- projected Adam ascent
    const float c1 = 1.f - powf(0.9f, (float)(it + 1)), c2 = 1.f - powf(0.999f, (float)(it + 1));
    for (int k = tid; k < d; k += kOptThreads) {
      const float g = gx[k];
      m1[k] = fmaf(0.9f, m1[k], 0.1f * g);
      m2[k] = fmaf(0.999f, m2[k], 0.001f * g * g);
      const float stp = a.lr * (m1[k] / c1) / (sqrtf(m2[k] / c2) + 1e-8f);
      xs[k] = fminf(fmaxf(xs[k] + stp, a.xlo[k]), a.xhi[k]);
    }
    __syncthreads();
  }
  for (int k = tid; k < d; k += kOptThreads) {
    a.X[((size_t)b * a.P + p) * d + k] = xs[k];
    if (a.grad) a.grad[((size_t)b * a.P + p) * d + k] = gx[k];
  }
  if (tid == 0) a.acq[(size_t)b * a.P + p] = val;
}

}  // namespace

int launch_acq_optimize(const Gp *gp, const float *lower, const float *upper, const int *K,
                        int box_cap, const float *eps, int S, const float *X0, int P,
                        const float *xlo, const float *xhi, int steps, float lr, float *X,
                        float *acq, float *grad, cudaStream_t s) {
  if (gp->m != 2 || gp->kern || gp->d > BOUTE_MAX_D) return BOUTE_ERR_UNSUPPORTED;
  OptArgs a;
  a.Wws = gp->Wws;
  a.xt = gp->xt;
  a.npad = gp->plan.npad;
  a.nxt = gp->plan.nxt;
  a.DP = gp->DP;
  a.n = gp->n;
  a.d = gp->d;
  a.m = gp->m;
  a.lower = lower;
  a.upper = upper;
  a.K = K;
  a.box_cap = box_cap;
  a.eps = eps;
  a.S = S;
  a.X0 = X0;
  a.xlo = xlo;
  a.xhi = xhi;
  a.P = P;
  a.steps = steps;
  a.lr = lr;
  a.X = X;
  a.acq = acq;
  a.grad = grad;
  const size_t smem = (4 * (size_t)gp->n + (size_t)gp->n * gp->d) * sizeof(float);
  if (smem > 200 * 1024) return BOUTE_ERR_UNSUPPORTED;
  prefer_shared(acqopt_kernel);
  cudaFuncSetAttribute(acqopt_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  launch_pdl(acqopt_kernel, dim3(P, gp->B), dim3(kOptThreads), smem, s, a);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
