// GP fit on the device: standardisation, kernel matrix, Cholesky factor,
// triangular inverse, alpha, and the prepacked tensor-core operands of the
// posterior contraction. All factor arithmetic is fp64 (Sec. 6: the paper's
// GP kernels run in double precision).
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace boute {

namespace {

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ double block_sum(double v, double *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double t = 0.0;
  for (int w = 0; w < nw; ++w) t += red[w];
  return t;
}

// ---- a0: Standardize (one block per (problem, objective)) --------------------
__global__ void standardize_kernel(const double *Y, int n, int m, double *Ys) {
  __shared__ double red[32];
  const int b = blockIdx.x / m, t = blockIdx.x % m;
  const double *y = Y + (size_t)b * n * m + t;
  double *ys = Ys + (size_t)b * n * m + t;
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += y[(size_t)i * m];
  const double mean = block_sum(s, red) / n;
  double ss = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    double z = y[(size_t)i * m] - mean;
    ss += z * z;
  }
  ss = block_sum(ss, red);
  double sd = n > 1 ? sqrt(ss / (n - 1)) : 1.0;
  if (!(sd >= 1e-8)) sd = 1.0;
  __syncthreads();  // every thread has read its inputs before (aliased) outputs land
  for (int i = threadIdx.x; i < n; i += blockDim.x) ys[(size_t)i * m] = (y[(size_t)i * m] - mean) / sd;
}

// ---- K = s2 M52(X, X) + noise I, per (problem, objective) --------------------
__global__ void kernel_matrix_kernel(const double *X, int n, int d, int m, const double *ls,
                                     const double *s2, const double *noise, double *Kall) {
  const int bt = blockIdx.z, b = bt / m;
  const int i = blockIdx.y * 16 + threadIdx.y, j = blockIdx.x * 16 + threadIdx.x;
  if (i >= n || j >= n) return;
  const double *xi = X + ((size_t)b * n + i) * d, *xj = X + ((size_t)b * n + j) * d;
  const double *l = ls + (size_t)bt * d;
  double r2 = 0.0;
  for (int t = 0; t < d; ++t) {
    double z = (xi[t] - xj[t]) / l[t];
    r2 += z * z;
  }
  const double r = sqrt(r2), sr = sqrt(5.0) * r;
  double k = s2[bt] * (1.0 + sr + 5.0 * r2 / 3.0) * exp(-sr);
  if (i == j) k += noise[bt];
  Kall[(size_t)bt * n * n + (size_t)i * n + j] = k;
}

// ---- scaled training inputs, 1/lengthscale and outputscale in fp32 -----------
__global__ void prep_kernel(const double *X, int n, int d, int m, int DP, int npad,
                            const double *ls, const double *s2, float *xt, float *invls,
                            float *s2f) {
  const int bt = blockIdx.y, b = bt / m;
  const double *l = ls + (size_t)bt * d;
  float *x = xt + (size_t)bt * npad * 2 * DP;
  const int total = npad * DP;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < total; e += gridDim.x * blockDim.x) {
    const int j = e / DP, t = e % DP;
    double v = (j < n && t < d) ? X[((size_t)b * n + j) * d + t] / l[t] : 0.0;
    float hi = (float)v, lo = (float)(v - (double)hi);
    const int c = j / BOUTE_KCHUNK, jj = j % BOUTE_KCHUNK;
    float *blk = x + (size_t)c * 2 * BOUTE_KCHUNK * DP;
    blk[jj * DP + t] = hi;
    blk[BOUTE_KCHUNK * DP + jj * DP + t] = lo;
  }
  if (blockIdx.x == 0) {
    for (int t = threadIdx.x; t < DP; t += blockDim.x) {
      double v = t < d ? 1.0 / l[t] : 0.0;
      float hi = (float)v;
      invls[(size_t)bt * 2 * DP + t] = hi;
      invls[(size_t)bt * 2 * DP + DP + t] = (float)(v - (double)hi);
    }
    if (threadIdx.x == 0) s2f[bt] = (float)s2[bt];
  }
}

// ---- right-looking Cholesky, one block per (problem, objective) --------------
// Column j: pivot sqrt, scale the column below it, rank-1 update of the
// trailing lower triangle (warp per row, lanes along the row). The matrix
// lives in shared memory when it fits, else in global memory (L2-resident).
template <bool SMEM>
__global__ void __launch_bounds__(512) chol_kernel(double *Kall, int n, int *status) {
  extern __shared__ double sm[];
  __shared__ int bad;
  __shared__ double piv;
  double *G = Kall + (size_t)blockIdx.x * n * n;
  double *A = SMEM ? sm : G;
  double *col = SMEM ? sm + (size_t)n * n : sm;
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5,
            nw = nthr >> 5;
  if (SMEM)
    for (int e = tid; e < n * n; e += nthr) A[e] = G[e];
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int j = 0; j < n; ++j) {
    if (tid == 0) {
      double p = A[(size_t)j * n + j];
      if (!(p > 0.0)) {
        bad = 1;
      } else {
        p = sqrt(p);
        A[(size_t)j * n + j] = p;
        piv = p;
      }
    }
    __syncthreads();
    if (bad) break;
    for (int i = j + 1 + tid; i < n; i += nthr) {
      double v = A[(size_t)i * n + j] / piv;
      A[(size_t)i * n + j] = v;
      col[i] = v;
    }
    __syncthreads();
    for (int i = j + 1 + warp; i < n; i += nw) {
      const double li = col[i];
      double *row = A + (size_t)i * n;
      for (int k = j + 1 + lane; k <= i; k += 32) row[k] -= li * col[k];
    }
    __syncthreads();
  }
  if (bad) {
    if (tid == 0) set_status(status, BOUTE_ERR_NOT_PD);
    return;
  }
  for (int e = tid; e < n * n; e += nthr) {
    const int i = e / n, k = e % n;
    G[e] = k <= i ? A[e] : 0.0;
  }
}

// ---- W = L^-1: one warp per column, forward substitution on e_j --------------
__global__ void trinv_kernel(const double *Lall, double *Wall, int n, const int *status) {
  extern __shared__ double wsm[];
  if (*status == BOUTE_ERR_NOT_PD) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int j = blockIdx.x * wpb + warp;
  const size_t bt = blockIdx.y;
  if (j >= n) return;
  const double *L = Lall + bt * n * n;
  double *W = Wall + bt * n * n;
  double *w = wsm + (size_t)warp * n;
  if (lane == 0) w[j] = 1.0 / L[(size_t)j * n + j];
  __syncwarp();
  for (int i = j + 1; i < n; ++i) {
    const double *Li = L + (size_t)i * n;
    double s = 0.0;
    for (int k = j + lane; k < i; k += 32) s += Li[k] * w[k];
    s = warp_sum(s);
    if (lane == 0) w[i] = -s / Li[i];
    __syncwarp();
  }
  for (int i = lane; i < n; i += 32) W[(size_t)i * n + j] = i >= j ? w[i] : 0.0;
}

// ---- alpha = W^T (W y) ------------------------------------------------------------
__global__ void alpha_kernel(const double *Wall, const double *Ys, int n, int m,
                             double *alpha_all, const int *status) {
  extern __shared__ double tv[];
  if (*status == BOUTE_ERR_NOT_PD) return;
  const int bt = blockIdx.x, b = bt / m, t = bt % m;
  const double *W = Wall + (size_t)bt * n * n;
  const double *y = Ys + (size_t)b * n * m + t;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (int i = warp; i < n; i += nw) {
    double s = 0.0;
    for (int k = lane; k <= i; k += 32) s += W[(size_t)i * n + k] * y[(size_t)k * m];
    s = warp_sum(s);
    if (lane == 0) tv[i] = s;
  }
  __syncthreads();
  for (int k = threadIdx.x; k < n; k += blockDim.x) {
    double s = 0.0;
    for (int i = k; i < n; ++i) s += W[(size_t)i * n + k] * tv[i];
    alpha_all[(size_t)bt * n + k] = s;
  }
}

// ---- operand images [L^-1 ; alpha^T] as tf32 hi/lo, swizzled -----------------
__global__ void pack_kernel(const double *Wall, const double *alpha_all, PostPlan plan,
                            float *bop, const int *status) {
  if (*status == BOUTE_ERR_NOT_PD) return;
  const size_t bt = blockIdx.y;
  const int n = plan.n;
  const double *W = Wall + bt * n * n;
  const double *al = alpha_all + bt * n;
  float *img = bop + bt * plan.image_floats;
  const long long total = (long long)plan.ncols * plan.npad;
  for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int g = (int)(e / plan.npad), k = (int)(e % plan.npad);
    const int p = g >> 8, c = k / BOUTE_KCHUNK;
    if (c >= plan.kc[p]) continue;
    double v = 0.0;
    if (k < n) {
      if (g < n) v = k <= g ? W[(size_t)g * n + k] : 0.0;
      else if (g == n) v = al[k];
    }
    const float hi = tf32_rna((float)v);
    const float lo = tf32_rna((float)(v - (double)hi));
    const int ncol = plan.ncol[p];
    float *blk = img + plan.off[p] + (long long)c * 2 * ncol * BOUTE_KCHUNK;
    const int o = sw128_off(g - plan.col0[p], k % BOUTE_KCHUNK);
    blk[o] = hi;
    blk[ncol * BOUTE_KCHUNK + o] = lo;
  }
}

}  // namespace

int launch_standardize(const double *Y, int B, int n, int m, double *Ys, cudaStream_t s) {
  standardize_kernel<<<B * m, 256, 0, s>>>(Y, n, m, Ys);
  count_launch();
  return last_launch_status();
}

int launch_fit(Gp *gp, const double *X, const double *Ys, const double *ls, const double *s2,
               const double *noise, cudaStream_t s) {
  const int n = gp->n, d = gp->d, m = gp->m, BM = gp->B * gp->m;
  cudaMemsetAsync(gp->status, 0, sizeof(int), s);  // a new fit starts with a clean status
  dim3 g1((n + 15) / 16, (n + 15) / 16, BM);
  kernel_matrix_kernel<<<g1, dim3(16, 16), 0, s>>>(X, n, d, m, ls, s2, noise, gp->K);
  prep_kernel<<<dim3(std::max(1, gp->plan.npad * gp->DP / 256), BM), 256, 0, s>>>(
      X, n, d, m, gp->DP, gp->plan.npad, ls, s2, gp->xt, gp->invls, gp->s2f);
  const size_t smem_chol = ((size_t)n * n + n) * sizeof(double);
  if (smem_chol <= 200 * 1024) {
    cudaFuncSetAttribute(chol_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem_chol);
    chol_kernel<true><<<BM, 512, smem_chol, s>>>(gp->K, n, gp->status);
  } else {
    chol_kernel<false><<<BM, 512, n * sizeof(double), s>>>(gp->K, n, gp->status);
  }
  const int wpb = 8;
  const size_t smem_inv = (size_t)wpb * n * sizeof(double);
  cudaFuncSetAttribute(trinv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_inv);
  trinv_kernel<<<dim3((n + wpb - 1) / wpb, BM), wpb * 32, smem_inv, s>>>(gp->K, gp->W, n,
                                                                          gp->status);
  alpha_kernel<<<BM, 256, n * sizeof(double), s>>>(gp->W, Ys, n, m, gp->alpha, gp->status);
  const long long tot = (long long)gp->plan.ncols * gp->plan.npad;
  pack_kernel<<<dim3((unsigned)std::min<long long>((tot + 255) / 256, 4096), BM), 256, 0, s>>>(
      gp->W, gp->alpha, gp->plan, gp->bop, gp->status);
  count_launch(6);
  return last_launch_status();
}

}  // namespace boute
