// The FP64 tier of the GP fit and posterior (Sec. 6 and Appendix C: the
// paper's MOBO runs its GP kernels in double precision): for a handle set to
// BOUTE_PREC_FP64, each fit also forms K in fp64, its Cholesky factor L, the
// inverse W = L^-1 and alpha = K^-1 y in fp64 (one block per problem-objective,
// K in shared memory), and boute_gp_posterior_fp64 evaluates
//   mean = k*^T alpha,  var = max(0, s2 - ||W k*||^2)
// in fp64 on the CUDA cores, one warp per candidate. GB300's fp64 rate is a
// small fraction of its fp32 rate, so this tier serves accuracy, not speed;
// it is limited to n <= 128 and the Matern-5/2 kernel.
#include <math.h>

#include "internal.h"

namespace boute {

namespace {

constexpr int kFit64Threads = 256;

__device__ __forceinline__ double matern52_d(double r2, double s2) {
  const double r = sqrt(r2);
  return s2 * (1.0 + 2.2360679774997896964 * r + (5.0 / 3.0) * r2) *
         exp(-2.2360679774997896964 * r);
}

// One block per (problem b, objective t): K (n x (n+1) fp64, lower triangle)
// in shared memory; right-looking Cholesky column by column (a pivot at or
// below 0 is BOUTE_ERR_NOT_PD); alpha by forward and back substitution; W =
// L^-1 in place, column by column from the last (the column's new entries
// need only the already inverted trailing block and the column of L itself).
// Writes W (n x n, lower, row-major), alpha (n) and X / l (n x d).
__global__ void __launch_bounds__(kFit64Threads) fit64_kernel(const double *X, const double *Ys,
                                                              const double *ls, const double *s2v,
                                                              const double *noise, int n, int d,
                                                              int m, double *W64, double *a64,
                                                              double *xs64, int *status) {
  extern __shared__ double K[];  // n x (n+1), then y / alpha (n)
  __shared__ int bad;
  const int bt = blockIdx.x, b = bt / m, t = bt % m, ld = n + 1;
  double *z = K + (size_t)n * ld;
  const double *x = X + (size_t)b * n * d, *l = ls + (size_t)bt * d;
  const double s2 = s2v[bt], nz = noise[bt];
  double *xs = xs64 + (size_t)bt * n * d;
  for (int e = threadIdx.x; e < n * d; e += blockDim.x) xs[e] = x[e] / l[e % d];
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
    const int i = e / n, j = e % n;
    if (j > i) continue;
    double r2 = 0.0;
    for (int k = 0; k < d; ++k) {
      const double df = xs[(size_t)i * d + k] - xs[(size_t)j * d + k];
      r2 = fma(df, df, r2);
    }
    K[(size_t)i * ld + j] = matern52_d(r2, s2) + (i == j ? nz : 0.0);
  }
  for (int i = threadIdx.x; i < n; i += blockDim.x) z[i] = Ys[((size_t)b * n + i) * m + t];
  __syncthreads();
  // Cholesky, column c: pivot, scaled column, trailing update (lower)
  for (int c = 0; c < n; ++c) {
    const double piv = K[(size_t)c * ld + c];
    if (!(piv > 0.0)) {
      if (threadIdx.x == 0) bad = 1;
      break;
    }
    const double lcc = sqrt(piv), inv = 1.0 / lcc;
    __syncthreads();
    if (threadIdx.x == 0) K[(size_t)c * ld + c] = lcc;
    for (int i = c + 1 + threadIdx.x; i < n; i += blockDim.x) K[(size_t)i * ld + c] *= inv;
    __syncthreads();
    const int rem = n - c - 1;
    for (int e = threadIdx.x; e < rem * rem; e += blockDim.x) {
      const int i = c + 1 + e / rem, j = c + 1 + e % rem;
      if (j <= i) K[(size_t)i * ld + j] = fma(-K[(size_t)i * ld + c], K[(size_t)j * ld + c],
                                              K[(size_t)i * ld + j]);
    }
    __syncthreads();
  }
  __syncthreads();
  if (bad) {
    if (threadIdx.x == 0) set_status(status, BOUTE_ERR_NOT_PD);
    return;
  }
  // alpha: L u = y (column-oriented), then L^T alpha = u (row-oriented)
  for (int c = 0; c < n; ++c) {
    if (threadIdx.x == 0) z[c] /= K[(size_t)c * ld + c];
    __syncthreads();
    const double zc = z[c];
    for (int i = c + 1 + threadIdx.x; i < n; i += blockDim.x)
      z[i] = fma(-K[(size_t)i * ld + c], zc, z[i]);
    __syncthreads();
  }
  for (int c = n - 1; c >= 0; --c) {
    if (threadIdx.x == 0) z[c] /= K[(size_t)c * ld + c];
    __syncthreads();
    const double zc = z[c];
    for (int i = threadIdx.x; i < c; i += blockDim.x) z[i] = fma(-K[(size_t)c * ld + i], zc, z[i]);
    __syncthreads();
  }
  for (int i = threadIdx.x; i < n; i += blockDim.x) a64[(size_t)bt * n + i] = z[i];
  // W = L^-1 in place: for j = n-1 .. 0, W_jj = 1 / L_jj and
  // W_ij = -W_jj sum_{k=j+1}^{i} W_ik L_kj (i > j), W_ik already final
  for (int j = n - 1; j >= 0; --j) {
    const double wjj = 1.0 / K[(size_t)j * ld + j];
    for (int i = j + 1 + threadIdx.x; i < n; i += blockDim.x) {
      double acc = 0.0;
      for (int k = j + 1; k <= i; ++k) acc = fma(K[(size_t)i * ld + k], K[(size_t)k * ld + j], acc);
      z[i] = -wjj * acc;  // (z is free after alpha)
    }
    __syncthreads();
    for (int i = j + 1 + threadIdx.x; i < n; i += blockDim.x) K[(size_t)i * ld + j] = z[i];
    if (threadIdx.x == 0) K[(size_t)j * ld + j] = wjj;
    __syncthreads();
  }
  double *Wout = W64 + (size_t)bt * n * n;
  for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
    const int i = e / n, j = e % n;
    Wout[e] = j <= i ? K[(size_t)i * ld + j] : 0.0;
  }
}

constexpr int kPost64Warps = 8;

// Candidates of one (problem, objective) per block-column y; one warp per
// candidate: lane j (mod 32) forms k*_j in fp64 into the warp's row of kb,
// lane i (mod 32) the rows i of v = W k*; mean = k*^T alpha.
__global__ void __launch_bounds__(32 * kPost64Warps) posterior64_kernel(
    const float *Xc, long long N, int n, int d, int m, const double *W64, const double *a64,
    const double *xs64, const double *ls, const double *s2v, double *mean, double *var) {
  extern __shared__ double sm64[];
  const int bt = blockIdx.y, b = bt / m, t = bt % m, ld = n + 1;
  double *Ws = sm64;                        // n x (n+1)
  double *al = Ws + (size_t)n * ld;         // n
  double *xs = al + n;                      // n x d
  double *kb = xs + (size_t)n * d;          // kPost64Warps x n
  const double *Wg = W64 + (size_t)bt * n * n;
  for (int e = threadIdx.x; e < n * n; e += blockDim.x) Ws[(size_t)(e / n) * ld + e % n] = Wg[e];
  for (int e = threadIdx.x; e < n; e += blockDim.x) al[e] = a64[(size_t)bt * n + e];
  for (int e = threadIdx.x; e < n * d; e += blockDim.x) xs[e] = xs64[(size_t)bt * n * d + e];
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const double s2 = s2v[bt];
  const double *l = ls + (size_t)bt * d;
  double *kw = kb + (size_t)warp * n;
  for (long long c = (long long)blockIdx.x * kPost64Warps + warp; c < N;
       c += (long long)gridDim.x * kPost64Warps) {
    const float *xc = Xc + ((size_t)b * N + c) * d;
    double mu = 0.0;
    for (int j = lane; j < n; j += 32) {
      double r2 = 0.0;
      for (int k = 0; k < d; ++k) {
        const double df = (double)xc[k] / l[k] - xs[(size_t)j * d + k];
        r2 = fma(df, df, r2);
      }
      const double kv = matern52_d(r2, s2);
      kw[j] = kv;
      mu = fma(kv, al[j], mu);
    }
    __syncwarp();
    double ss = 0.0;
    for (int i = lane; i < n; i += 32) {
      const double *wr = Ws + (size_t)i * ld;
      double v = 0.0;
      for (int j = 0; j <= i; ++j) v = fma(wr[j], kw[j], v);
      ss = fma(v, v, ss);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      mu += __shfl_xor_sync(0xffffffffu, mu, o);
      ss += __shfl_xor_sync(0xffffffffu, ss, o);
    }
    if (lane == 0) {
      const size_t o = ((size_t)b * m + t) * N + c;
      mean[o] = mu;
      const double vv = s2 - ss;
      var[o] = vv > 0.0 ? vv : 0.0;
    }
    __syncwarp();
  }
}

}  // namespace

size_t fit64_smem_bytes(int n) { return ((size_t)n * (n + 1) + n) * sizeof(double); }
size_t post64_smem_bytes(int n, int d) {
  return ((size_t)n * (n + 1) + n + (size_t)n * d + (size_t)kPost64Warps * n) * sizeof(double);
}

int launch_fit64(Gp *gp, const double *X, const double *Ys, const double *ls, const double *s2,
                 const double *noise, cudaStream_t s) {
  const size_t smem = fit64_smem_bytes(gp->n);
  if (cudaFuncSetAttribute(fit64_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return last_launch_status();
  fit64_kernel<<<gp->B * gp->m, kFit64Threads, smem, s>>>(X, Ys, ls, s2, noise, gp->n, gp->d,
                                                          gp->m, gp->W64, gp->a64, gp->xs64,
                                                          gp->status);
  count_launch();
  return last_launch_status();
}

int launch_posterior64(const Gp *gp, const float *Xc, long long N, double *mean, double *var,
                       cudaStream_t s) {
  if (N <= 0) return BOUTE_OK;
  const size_t smem = post64_smem_bytes(gp->n, gp->d);
  if (cudaFuncSetAttribute(posterior64_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return last_launch_status();
  const long long per = (N + kPost64Warps - 1) / kPost64Warps;
  const unsigned gx = (unsigned)std::max(1LL, std::min<long long>(per, 2LL * num_sms()));
  posterior64_kernel<<<dim3(gx, gp->B * gp->m), 32 * kPost64Warps, smem, s>>>(
      Xc, N, gp->n, gp->d, gp->m, gp->W64, gp->a64, gp->xs64, gp->ls64, gp->s2_64, mean, var);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
