// Hyperparameter learning by maximising the GP's log marginal likelihood
// (Sec. 6: the ARD lengthscales and outputscale are learned jointly by
// maximising the marginal likelihood; all kernels in double precision).
//
// One block per (problem, objective, restart) runs the whole optimisation:
// per Adam step it builds K = s2 M52(X, X) + noise I in fp64, factors it in
// place (right-looking Cholesky), inverts the factor in place, forms K^-1 in
// place, alpha = K^-1 y, the log likelihood and its gradient with respect to
// theta = (log l_1 .. log l_d, log s2, log noise),
//   d log p / d theta_q = 1/2 sum_ij (alpha_i alpha_j - K^-1_ij) dK_ij / dtheta_q,
// then takes a bias-corrected Adam ascent step and clamps theta to its
// bounds. The lower triangle of the n x n workspace holds K, then L, then
// L^-1, then K^-1; the upper triangle keeps exp(-sqrt5 r_ij) for the gradient.
// The workspace is in shared memory when it fits, else in global memory
// (one slice per block, L2-resident).
#include <math.h>

#include "internal.h"

namespace boute {

namespace {

constexpr int kLearnThreads = 256;
constexpr int kLearnWarps = kLearnThreads / 32;
constexpr int kLearnRows = 8;  // rows of K^-1 formed per pass
constexpr double kSqrt5d = 2.23606797749978969641;
constexpr double kSqrt3d = 1.73205080756887729353;
constexpr double kLog2Pi = 1.83787706640934548356;

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Entry e of a lower triangle (diagonal included, row by row) -> (i, j).
__device__ __forceinline__ void tri_index(int e, int &i, int &j) {
  int r = (int)((sqrtf(8.f * (float)e + 1.f) - 1.f) * 0.5f);
  while (r * (r + 1) / 2 > e) --r;
  while ((r + 1) * (r + 2) / 2 <= e) ++r;
  i = r;
  j = e - r * (r + 1) / 2;
}

__device__ __forceinline__ double clamp_d(double v, double lo, double hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

// theta_q clamped to its bound: q < d log l, d log s2, d + 1 log noise, then
// (composite kernel) d + 2 log s2_c, d + 3 log s2_x, d + 4 beta
__device__ __forceinline__ double clamp_param(int q, int d, double v) {
  if (q < d) return clamp_d(v, BOUTE_LOG_LS_MIN, BOUTE_LOG_LS_MAX);
  if (q == d) return clamp_d(v, BOUTE_LOG_S2_MIN, BOUTE_LOG_S2_MAX);
  if (q == d + 1) return clamp_d(v, BOUTE_LOG_NOISE_MIN, BOUTE_LOG_NOISE_MAX);
  if (q < d + 4) return clamp_d(v, BOUTE_LOG_SC_MIN, BOUTE_LOG_SC_MAX);
  return clamp_d(v, BOUTE_BETA_MIN, BOUTE_BETA_MAX);
}

// Row stride of the n x n workspace: odd, so that a column's 64-bit entries
// fall in different shared-memory banks.
__host__ __device__ inline int learn_ld(int n) { return n | 1; }

// Doubles of one block's workspace: A (n x ld), X (n x d), y, alpha, tmp,
// 1 / L_jj (n each), tmp2 (kLearnRows rows of K^-1), and for the composite
// kernel <s, c_i> and w_i (n each).
__host__ __device__ inline size_t learn_ws_doubles(int n, int d) {
  return (size_t)n * learn_ld(n) + (size_t)n * d + 6 * (size_t)n + (size_t)kLearnRows * n;
}

constexpr int kMaxP = BOUTE_MAX_D + 5;  // parameters of the composite kernel

// COMP: the composite kernel (routing features [0, dtau), preference entries
// pref: B x m x (d - dtau)), theta extended by (log s2_c, log s2_x, beta):
//   K = s2 k52(r_t) + s2_c w_i w_j k32(r_c) + s2_x k52 k32 + noise I,
//   dK/dlog l_q = (5/3)(1 + sqrt5 r_t) e^(-sqrt5 r_t) z_q^2 (s2 + s2_x k32)  (routing)
//               = 3 e^(-sqrt3 r_c) z_q^2 (s2_c w_i w_j + s2_x k52)        (deployment)
//   dK/dlog s2_c = s2_c w_i w_j k32, dK/dlog s2_x = s2_x k52 k32,
//   dK/dbeta = s2_c w_i w_j k32 (<s, c_i> + <s, c_j>).
template <bool COMP>
__global__ void __launch_bounds__(kLearnThreads) learn_kernel(
    const double *X, const double *Ys, int n, int d, int m, int R, const double *theta0,
    int iters, double lr, double *theta_out, double *mll_out, double *grad_out, double *ws,
    int use_smem, int dtau, const double *pref) {
  extern __shared__ __align__(16) double lsm[];
  __shared__ double th[kMaxP], m1[kMaxP], m2[kMaxP];
  __shared__ double il[BOUTE_MAX_D], red[kLearnWarps][kMaxP];
  __shared__ double logdet, mll_s;
  __shared__ int bad;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int blk = blockIdx.x, bt = blk / R, b = bt / m, t = bt % m;
  const int P = d + (COMP ? 5 : 2), ld = learn_ld(n), dc = d - dtau;
  double *A = use_smem ? lsm : ws + (size_t)blk * learn_ws_doubles(n, d);
  double *xs = A + (size_t)n * ld, *yv = xs + (size_t)n * d, *av = yv + n, *tmp = av + n, *dinv = tmp + n,
         *tmp2 = dinv + n, *pc = tmp2 + (size_t)kLearnRows * n, *wv = pc + n;
  for (int e = tid; e < n * d; e += kLearnThreads) xs[e] = X[(size_t)b * n * d + e];
  for (int i = tid; i < n; i += kLearnThreads) yv[i] = Ys[((size_t)b * n + i) * m + t];
  const double *th0 = theta0 + (size_t)blk * P;
  if (tid < P) {
    th[tid] = clamp_param(tid, d, th0[tid]);
    m1[tid] = 0.0;
    m2[tid] = 0.0;
  }
  if (COMP) {  // <s, c_i> of the training points (s fixed)
    __syncthreads();
    const double *pb = pref + (size_t)bt * dc;
    for (int i = tid; i < n; i += kLearnThreads) {
      double e = 0.0;
      for (int k = 0; k < dc; ++k) e = fma(pb[k], xs[(size_t)i * d + dtau + k], e);
      pc[i] = e;
    }
  }
  double b1t = 1.0, b2t = 1.0;
  __syncthreads();

  for (int it = 0; it <= iters; ++it) {
    const bool last = it == iters;
    const bool want_grad = !last || grad_out != nullptr;
    // ---- K (lower) and exp(-sqrt5 r) (upper) at theta
    if (tid < d) il[tid] = exp(-th[tid]);
    if (tid == 0) bad = 0;
    if (COMP)
      for (int i = tid; i < n; i += kLearnThreads) wv[i] = exp(th[d + 4] * pc[i]);
    __syncthreads();
    const double s2 = exp(th[d]), nz = exp(th[d + 1]);
    const double s2c = COMP ? exp(th[d + 2]) : 0.0, s2x = COMP ? exp(th[d + 3]) : 0.0;
    const int npair = n * (n + 1) / 2;  // pairs i >= j, one thread each
    for (int e = tid; e < npair; e += kLearnThreads) {
      int i, j;
      tri_index(e, i, j);
      if (COMP) {  // (the gradient recomputes the exponentials)
        double rt2 = 0.0, rc2 = 0.0;
        for (int q = 0; q < d; ++q) {
          const double z = (xs[i * d + q] - xs[j * d + q]) * il[q];
          if (q < dtau) rt2 = fma(z, z, rt2);
          else rc2 = fma(z, z, rc2);
        }
        const double st = kSqrt5d * sqrt(rt2), sc = kSqrt3d * sqrt(rc2);
        const double k52 = (1.0 + st + 5.0 * rt2 / 3.0) * exp(-st), k32 = (1.0 + sc) * exp(-sc);
        A[(size_t)i * ld + j] =
            s2 * k52 + s2c * wv[i] * wv[j] * k32 + s2x * k52 * k32 + (i == j ? nz : 0.0);
        continue;
      }
      double r2 = 0.0;
      for (int q = 0; q < d; ++q) {
        const double z = (xs[i * d + q] - xs[j * d + q]) * il[q];
        r2 = fma(z, z, r2);
      }
      const double rr = sqrt(r2), sr = kSqrt5d * rr, ex = exp(-sr);
      A[(size_t)i * ld + j] = s2 * (1.0 + sr + 5.0 * r2 / 3.0) * ex + (i == j ? nz : 0.0);
      if (i != j) A[(size_t)j * ld + i] = ex;
    }
    // ---- Cholesky in place (lower), column by column
    for (int j = 0; j < n; ++j) {
      __syncthreads();
      const double djj = A[(size_t)j * ld + j];
      if (!(djj > 0.0)) {  // not positive definite (every thread sees the same value)
        if (tid == 0) bad = 1;
        break;
      }
      // one reciprocal square root on the column's critical path
      const double inv = rsqrt(djj), Ljj = djj * inv;
      for (int i = j + 1 + tid; i < n; i += kLearnThreads) A[(size_t)i * ld + j] *= inv;
      __syncthreads();
      // (the diagonal entry is replaced only now: every thread has read it)
      if (tid == 0) A[(size_t)j * ld + j] = Ljj;
      for (int i = j + 1 + warp; i < n; i += kLearnWarps) {
        const double lij = A[(size_t)i * ld + j];
        for (int k = j + 1 + lane; k <= i; k += 32)
          A[(size_t)i * ld + k] = fma(-lij, A[(size_t)k * ld + j], A[(size_t)i * ld + k]);
      }
    }
    __syncthreads();
    if (bad) break;  // keeps theta; the evaluation after the loop reports NaN
    // log det K = 2 sum_j log L_jj (off the factorisation's critical path),
    // and the reciprocals of the diagonal for the inversion
    if (warp == 0) {
      double s = 0.0;
      for (int j = lane; j < n; j += 32) s += log(A[(size_t)j * ld + j]);
      s = warp_sum_d(s);
      if (lane == 0) logdet = s;
    }
    for (int j = tid; j < n; j += kLearnThreads) dinv[j] = 1.0 / A[(size_t)j * ld + j];
    __syncthreads();
    // ---- L^-1 in place by forward substitution of L X = I, right-looking:
    // step k finishes row k of X (row k of B divided by L_kk) and subtracts
    // L_ik times it from the rows i > k of B (B = I initially). Entry (i, c)
    // holds L_ic until step c has used it, then B_ic, then X_ic.
    for (int k = 0; k < n; ++k) {
      const double ikk = dinv[k];
      for (int i = k + 1 + tid; i < n; i += kLearnThreads) tmp[i] = A[(size_t)i * ld + k];
      __syncthreads();  // column k of L saved; every thread has read L_kk
      for (int c = tid; c <= k; c += kLearnThreads)
        A[(size_t)k * ld + c] = c == k ? ikk : A[(size_t)k * ld + c] * ikk;
      __syncthreads();
      const int w = k + 1;  // entries per row to update: columns 0 .. k
      for (int e = tid; e < (n - k - 1) * w; e += kLearnThreads) {
        const int i = k + 1 + e / w, c = e - (e / w) * w;
        const double xkc = A[(size_t)k * ld + c];
        A[(size_t)i * ld + c] = c == k ? -tmp[i] * xkc : fma(-tmp[i], xkc, A[(size_t)i * ld + c]);
      }
      __syncthreads();  // tmp is rewritten by the next step
    }
    // ---- K^-1 = X^T X in place (X = L^-1 lower), kLearnRows rows at a time:
    // entry (i, j <= i) is sum_{k >= i} X_ki X_kj, which needs only rows >= i
    // of X, so a batch of rows is computed into tmp2 and written back after
    __syncthreads();
    for (int i0 = 0; i0 < n; i0 += kLearnRows) {
      const int i1 = min(n, i0 + kLearnRows);
      const int cnt = (i1 - i0) * i0 + (i1 - i0) * (i1 - i0 + 1) / 2;  // entries j <= i
      for (int e = tid; e < cnt; e += kLearnThreads) {
        // entry e -> (i, j): rows of i0 + 1, i0 + 2, ... entries
        int i = i0, base = 0;
        while (base + i + 1 <= e) {
          base += i + 1;
          ++i;
        }
        const int j = e - base;
        double s = 0.0;
        for (int k = i; k < n; ++k) s = fma(A[(size_t)k * ld + i], A[(size_t)k * ld + j], s);
        tmp2[e] = s;
      }
      __syncthreads();
      for (int e = tid; e < cnt; e += kLearnThreads) {
        int i = i0, base = 0;
        while (base + i + 1 <= e) {
          base += i + 1;
          ++i;
        }
        A[(size_t)i * ld + (e - base)] = tmp2[e];
      }
      __syncthreads();
    }
    // ---- alpha = K^-1 y and the log likelihood
    for (int i = warp; i < n; i += kLearnWarps) {
      double s = 0.0;
      for (int j = lane; j < n; j += 32) {
        const double kij = j <= i ? A[(size_t)i * ld + j] : A[(size_t)j * ld + i];
        s = fma(kij, yv[j], s);
      }
      s = warp_sum_d(s);
      if (lane == 0) av[i] = s;
    }
    __syncthreads();
    if (tid < 32) {
      double s = 0.0;
      for (int i = lane; i < n; i += 32) s = fma(yv[i], av[i], s);
      s = warp_sum_d(s);
      if (lane == 0) mll_s = -0.5 * s - logdet - 0.5 * (double)n * kLog2Pi;
    }
    if (!want_grad) break;
    // ---- gradient: pairs i >= j (an off-diagonal pair stands for two
    // entries); per pair f = s2 (5/3) (1 + sqrt5 r) e^(-sqrt5 r) multiplies
    // (dx_q / l_q)^2 in the lengthscale terms
    double g[BOUTE_MAX_D], gs2 = 0.0, gnz = 0.0, gsc = 0.0, gsx = 0.0, gbe = 0.0;
#pragma unroll
    for (int q = 0; q < BOUTE_MAX_D; ++q) g[q] = 0.0;
    for (int e = tid; e < npair; e += kLearnThreads) {
      int i, j;
      tri_index(e, i, j);
      const double Q = (i == j ? 0.5 : 1.0) * (av[i] * av[j] - A[(size_t)i * ld + j]);
      const double *xi = xs + (size_t)i * d, *xj = xs + (size_t)j * d;
      if (COMP) {
        double rt2 = 0.0, rc2 = 0.0;
        for (int q = 0; q < d; ++q) {
          const double z = (xi[q] - xj[q]) * il[q];
          if (q < dtau) rt2 = fma(z, z, rt2);
          else rc2 = fma(z, z, rc2);
        }
        const double st = kSqrt5d * sqrt(rt2), sc = kSqrt3d * sqrt(rc2);
        const double e5 = exp(-st), e3 = exp(-sc);
        const double k52 = (1.0 + st + 5.0 * rt2 / 3.0) * e5, k32 = (1.0 + sc) * e3;
        const double ww = wv[i] * wv[j];
        const double ft = Q * (5.0 / 3.0) * (1.0 + st) * e5 * (s2 + s2x * k32);
        const double fc = Q * 3.0 * e3 * (s2c * ww + s2x * k52);
#pragma unroll
        for (int q = 0; q < BOUTE_MAX_D; ++q) {
          if (q < d) {
            const double z = (xi[q] - xj[q]) * il[q];
            g[q] = fma(q < dtau ? ft : fc, z * z, g[q]);
          }
        }
        gs2 = fma(Q, s2 * k52, gs2);
        if (i == j) gnz = fma(Q, nz, gnz);
        const double tc = Q * s2c * ww * k32;
        gsc += tc;
        gsx = fma(Q, s2x * k52 * k32, gsx);
        gbe = fma(tc, pc[i] + pc[j], gbe);
        continue;
      }
      double r2 = 0.0;
      for (int q = 0; q < d; ++q) {
        const double z = (xi[q] - xj[q]) * il[q];
        r2 = fma(z, z, r2);
      }
      const double rr = sqrt(r2), sr = kSqrt5d * rr;
      const double ex = i == j ? 1.0 : A[(size_t)j * ld + i];
      const double Qf = Q * s2 * (5.0 / 3.0) * (1.0 + sr) * ex;
#pragma unroll
      for (int q = 0; q < BOUTE_MAX_D; ++q) {
        if (q < d) {
          const double z = (xi[q] - xj[q]) * il[q];
          g[q] = fma(Qf, z * z, g[q]);
        }
      }
      gs2 = fma(Q, s2 * (1.0 + sr + 5.0 * r2 / 3.0) * ex, gs2);
      if (i == j) gnz = fma(Q, nz, gnz);
    }
    // block sums of the d + 2 components (the pair sums already carry the 1/2)
#pragma unroll
    for (int q = 0; q < BOUTE_MAX_D; ++q) {
      if (q < d) {
        const double v = warp_sum_d(g[q]);
        if (lane == 0) red[warp][q] = v;
      }
    }
    {
      const double a = warp_sum_d(gs2), c = warp_sum_d(gnz);
      if (lane == 0) {
        red[warp][d] = a;
        red[warp][d + 1] = c;
      }
      if (COMP) {
        const double u = warp_sum_d(gsc), v2 = warp_sum_d(gsx), w2 = warp_sum_d(gbe);
        if (lane == 0) {
          red[warp][d + 2] = u;
          red[warp][d + 3] = v2;
          red[warp][d + 4] = w2;
        }
      }
    }
    __syncthreads();
    if (tid < P) {
      double v = 0.0;
      for (int w = 0; w < kLearnWarps; ++w) v += red[w][tid];
      if (last) {
        grad_out[(size_t)blk * P + tid] = v;
      } else {
        // Adam ascent step, bias-corrected moments, then the bounds
        b1t *= BOUTE_ADAM_B1;
        b2t *= BOUTE_ADAM_B2;
        m1[tid] = BOUTE_ADAM_B1 * m1[tid] + (1.0 - BOUTE_ADAM_B1) * v;
        m2[tid] = BOUTE_ADAM_B2 * m2[tid] + (1.0 - BOUTE_ADAM_B2) * v * v;
        const double mh = m1[tid] / (1.0 - b1t), vh = m2[tid] / (1.0 - b2t);
        th[tid] = clamp_param(tid, d, th[tid] + lr * mh / (sqrt(vh) + BOUTE_ADAM_EPS));
      }
    }
    __syncthreads();
  }
  __syncthreads();
  if (tid < P) theta_out[(size_t)blk * P + tid] = th[tid];
  if (tid == 0) mll_out[blk] = bad ? nan("") : mll_s;
  if (bad && grad_out && tid < P) grad_out[(size_t)blk * P + tid] = nan("");
}

}  // namespace

size_t learn_smem_limit() { return 200 * 1024; }

// dtau, pref: the composite kernel (pref null: the Matern-5/2 kernel)
int launch_learn(const double *X, const double *Ys, int B, int n, int d, int m,
                 const double *theta0, int R, int iters, double lr, double *theta, double *mll,
                 double *grad, int dtau, const double *pref, cudaStream_t s) {
  const size_t per = learn_ws_doubles(n, d) * sizeof(double);
  const int blocks = B * m * R;
  const bool smem = per <= learn_smem_limit();
  double *ws = nullptr;
  if (!smem && cudaMallocAsync((void **)&ws, per * blocks, s) != cudaSuccess) {
    cudaGetLastError();
    return BOUTE_ERR_OOM;
  }
  auto go = [&](auto kern) {
    if (smem) {
      prefer_shared(kern);
      if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)per) !=
          cudaSuccess)
        return;
    }
    kern<<<blocks, kLearnThreads, smem ? per : 0, s>>>(X, Ys, n, d, m, R, theta0, iters, lr,
                                                       theta, mll, grad, ws, smem ? 1 : 0, dtau,
                                                       pref);
  };
  if (pref) go(learn_kernel<true>);
  else go(learn_kernel<false>);
  count_launch();
  const int st = last_launch_status();
  if (ws) cudaFreeAsync(ws, s);
  return st;
}

}  // namespace boute
