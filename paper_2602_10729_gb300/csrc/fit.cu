// GP fit on the device (Sec. 5.2, one exact GP per objective; Sec. 6,
// Matern-5/2 ARD kernel with outputscale on standardised outcomes):
// standardisation, kernel matrix, Cholesky factor, triangular inverse, alpha,
// and the prepacked tensor-core operands of the posterior contraction. The
// kernel matrix is formed in fp64 and kept as an fp32 pair; the factor and its
// inverse are fp32, and alpha is refined against the fp64-accurate matrix
// with double-float residuals (the paper runs its GP kernels in double
// precision, Appendix C; fp64 throughput is low on this part).
#include <math.h>

#include <algorithm>

#include <type_traits>

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

// ---- Standardize (one block per (problem, objective)) --------------------
// (codes: outcome transforms, objective_code)
__global__ void standardize_kernel(const double *Y, int n, int m, int codes, double *Ys) {
  __shared__ double red[32];
  const int b = blockIdx.x / m, t = blockIdx.x % m;
  const int code = objective_code(codes, t);
  const double *y = Y + (size_t)b * n * m + t;
  double *ys = Ys + (size_t)b * n * m + t;
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += outcome_transform(y[(size_t)i * m], code);
  const double mean = block_sum(s, red) / n;
  double ss = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    double z = outcome_transform(y[(size_t)i * m], code) - mean;
    ss += z * z;
  }
  ss = block_sum(ss, red);
  double sd = n > 1 ? sqrt(ss / (n - 1)) : 1.0;
  if (!(sd >= 1e-8)) sd = 1.0;
  const double isd = 1.0 / sd;  // one division; fp64 divides are slow on this part
  __syncthreads();  // every thread has read its inputs before (aliased) outputs land
  for (int i = threadIdx.x; i < n; i += blockDim.x)
    ys[(size_t)i * m] = (outcome_transform(y[(size_t)i * m], code) - mean) * isd;
}

// ---- fit set-up, one launch: K = s2 M52(X, X) + noise I and the side input --
// Blocks [0, nkt) of problem-objective bt compute K in fp64, one half (16 x 8)
// of a 16 x 16 tile on or below the diagonal per block of 128 threads, each
// value written to both (i, j) and (j, i), stored as an fp32 pair (hi = K
// rounded, lo = K - hi): the factorisation works on hi, the refinement of
// alpha on hi + lo. (The set-up is bound by fp64 throughput: the lower
// triangle alone, spread over as many SMs as possible.) The remaining blocks
// write the posterior's side input: scaled training inputs x / l as fp32
// hi/lo pairs (dimension-major per 32-point chunk), and in every chunk the
// objective's 1/l (hi, lo) and outputscale. Block 0 of the first problem
// clears the fit status.
// Composite kernel (kp != null: [s2_c, s2_x, beta, s_0 .. s_{d-1}] of this
// problem-objective, s_k = 0 for the routing features [0, dtau)), Sec. 5.2
// "Additive kernels" and S5 as Sec. 6 assembles them:
//   k = s2 k52(r_t) + s2_c w_i w_j k32(r_c) + s2_x k52(r_t) k32(r_c),
// r_t over the routing features, r_c over the deployment features,
// w = exp(beta sum_k s_k x_k). Its side input holds, in place of the
// coordinates' lo parts, the training points' weights w_j and beta s_k, and
// s2_c, s2_x, dtau after the outputscale.
constexpr int kSetupThreads = 128;
__host__ __device__ inline int kmat_units(int n) {
  const int tn = (n + 15) / 16;
  return tn * (tn + 1);  // tiles on or below the diagonal, two halves each
}
// COMP: the composite kernel (kp its parameters); the Matern-5/2
// instantiation carries none of its code.
template <bool COMP>
__device__ void kmat_tile(const double *X, int n, int d, int b, const double *l, double s2,
                          double noise, int unit, float *Kh, float *Kl, double *il,
                          const double *kp, int dtau) {
  for (int t = threadIdx.x; t < d; t += blockDim.x) il[t] = 1.0 / l[t];
  __syncthreads();
  const int tile = unit >> 1, half = unit & 1;
  int ti = (int)((sqrtf(8.f * tile + 1.f) - 1.f) * 0.5f);  // tile = ti (ti + 1) / 2 + tj
  while (ti * (ti + 1) / 2 > tile) --ti;
  while ((ti + 1) * (ti + 2) / 2 <= tile) ++ti;
  const int tj = tile - ti * (ti + 1) / 2;
  const int i = ti * 16 + threadIdx.x / 8, j = tj * 16 + half * 8 + threadIdx.x % 8;
  if (i >= n || j >= n) return;
  const double *xi = X + ((size_t)b * n + i) * d, *xj = X + ((size_t)b * n + j) * d;
  double r2 = 0.0, r2c = 0.0;
  const int dt = COMP ? dtau : d;
  for (int t = 0; t < dt; ++t) {
    const double z = (xi[t] - xj[t]) * il[t];
    r2 = fma(z, z, r2);
  }
  if (COMP) {
    for (int t = dt; t < d; ++t) {
      const double z = (xi[t] - xj[t]) * il[t];
      r2c = fma(z, z, r2c);
    }
  }
  const double r = sqrt(r2), sr = sqrt(5.0) * r;
  double k;
  if (!COMP) {
    k = s2 * (1.0 + sr + 5.0 * r2 / 3.0) * exp(-sr);
  } else {
    const double k52 = (1.0 + sr + 5.0 * r2 / 3.0) * exp(-sr);
    const double sc = sqrt(3.0) * sqrt(r2c), k32 = (1.0 + sc) * exp(-sc);
    double ei = 0.0, ej = 0.0;
    for (int t = dtau; t < d; ++t) {
      ei = fma(kp[3 + t], xi[t], ei);
      ej = fma(kp[3 + t], xj[t], ej);
    }
    k = s2 * k52 + kp[0] * exp(kp[2] * (ei + ej)) * k32 + kp[1] * k52 * k32;
  }
  if (i == j) k += noise;
  const float kh = (float)k, kl = (float)(k - (double)kh);
  Kh[(size_t)i * n + j] = kh;
  Kl[(size_t)i * n + j] = kl;
  if (i != j) {  // (the same value: the squared differences are symmetric)
    Kh[(size_t)j * n + i] = kh;
    Kl[(size_t)j * n + i] = kl;
  }
}

template <bool COMP>
__device__ void prep_part(const double *X, int n, int d, int b, int DP, int npad,
                          const double *l, double s2, double noise, float *x, int blk, int nblk,
                          const double *kp, int dtau) {
  const int cf = xt_chunk_floats(DP);
  const int total = npad * DP;
  for (int e = blk * blockDim.x + threadIdx.x; e < total; e += nblk * blockDim.x) {
    const int j = e / DP, t = e % DP;
    const double cs = (COMP && t >= dtau) ? kCoordScale32 : kCoordScale52;
    double v = (j < n && t < d) ? X[((size_t)b * n + j) * d + t] / l[t] * cs : 0.0;
    float hi = (float)v, lo = (float)(v - (double)hi);
    const int c = j / BOUTE_KCHUNK, jj = j % BOUTE_KCHUNK;
    float *q = x + (size_t)c * cf;  // dimension-major: [DP][32] hi, [DP][32] lo
    q[t * BOUTE_KCHUNK + jj] = hi;
    if (!COMP) q[BOUTE_KCHUNK * DP + t * BOUTE_KCHUNK + jj] = lo;
  }
  if (COMP) {  // composite kernel: w_j (row 0 of the lo block), beta s_k (row 1)
    for (int e = blk * blockDim.x + threadIdx.x; e < npad; e += nblk * blockDim.x) {
      double ej = 0.0;
      if (e < n)
        for (int t = dtau; t < d; ++t) ej = fma(kp[3 + t], X[((size_t)b * n + e) * d + t], ej);
      x[(size_t)(e / BOUTE_KCHUNK) * cf + BOUTE_KCHUNK * DP + e % BOUTE_KCHUNK] =
          e < n ? (float)exp(kp[2] * ej) : 0.f;
    }
    for (int e = blk * blockDim.x + threadIdx.x; e < (npad / BOUTE_KCHUNK) * DP;
         e += nblk * blockDim.x) {
      const int c = e / DP, k = e % DP;
      x[(size_t)c * cf + BOUTE_KCHUNK * DP + BOUTE_KCHUNK + k] =
          (k >= dtau && k < d) ? (float)(kp[2] * kp[3 + k]) : 0.f;
    }
  }
  const int po = xt_param_offset(DP), nch = npad / BOUTE_KCHUNK, np = 2 * DP + 8;
  for (int e = blk * blockDim.x + threadIdx.x; e < nch * np; e += nblk * blockDim.x) {
    const int c = e / np, k = e % np;
    float v = 0.f;
    // the coordinates' scale over l (hi, lo)
    if (k < DP) v = k < d ? (float)(((COMP && k >= dtau) ? kCoordScale32 : kCoordScale52) / l[k]) : 0.f;
    else if (k < 2 * DP) {
      const int t = k - DP;
      if (t < d) {
        const double iv = ((COMP && t >= dtau) ? kCoordScale32 : kCoordScale52) / l[t];
        v = (float)(iv - (double)(float)iv);
      }
    } else if (k == 2 * DP + kParS2) v = (float)s2;
    else if (COMP && k == 2 * DP + kParS2c) v = (float)kp[0];
    else if (COMP && k == 2 * DP + kParS2x) v = (float)kp[1];
    else if (COMP && k == 2 * DP + kParDtau) v = (float)dtau;
    else if (k == 2 * DP + kParEW)  // the prior variance bounds K's diagonal from above
      v = (float)w_scale_exp(noise, COMP ? s2 + kp[0] + kp[1] : s2);
    x[(size_t)c * cf + po + k] = v;
  }
}

template <bool COMP>
__global__ void __launch_bounds__(kSetupThreads) fit_setup_kernel(
    const double *X, int n, int d, int m, int DP, int npad, const double *ls, const double *s2,
    const double *noise, float *Kh_all, float *Kl_all, float *xt, float *s2f, int nkt, int nprep,
    int early_trigger, int *status, const double *kpar, int dtau) {
  __shared__ double il[BOUTE_MAX_D];
  const int bt = blockIdx.y, b = bt / m;
  if (early_trigger) pdl_trigger();  // the whole grid is resident: the fit may launch now
  const double *l = ls + (size_t)bt * d;
  const double *kp = COMP ? kpar + (size_t)bt * (3 + d) : nullptr;
  if (blockIdx.x == 0 && bt == 0 && threadIdx.x == 0) *status = BOUTE_OK;
  if ((int)blockIdx.x < nkt) {
    kmat_tile<COMP>(X, n, d, b, l, s2[bt], noise[bt], blockIdx.x, Kh_all + (size_t)bt * n * n,
                    Kl_all + (size_t)bt * n * n, il, kp, dtau);
  } else {
    float *x = xt + (size_t)bt * (npad / BOUTE_KCHUNK) * xt_chunk_floats(DP);
    prep_part<COMP>(X, n, d, b, DP, npad, l, s2[bt], noise[bt], x, blockIdx.x - nkt, nprep, kp,
                    dtau);
    // the prior variance's constant part (composite: s2 + s2_x; the
    // posterior adds s2_c w(x)^2)
    if (blockIdx.x == nkt && threadIdx.x == 0) s2f[bt] = (float)(COMP ? s2[bt] + kp[1] : s2[bt]);
  }
}

// The fp16 hi/lo operand images of W = L^-1 scaled by 2^e_W (see PostPlan):
// the pair of elements (g, k), (g, k + 1) of W (row g = output column, k
// even), zero above the diagonal and beyond n. Returns false if a scaled
// element reaches the fp16 range (W beyond four times its bound 1/sigma_n:
// the fp32 factor is numerically singular).
__device__ __forceinline__ bool pack_pair(const float *wrow, int g, int k, const PostPlan &plan,
                                          float scale, uint16_t *img) {
  const int n = plan.n;
  const float v0 = (k < n && g < n && k <= g) ? wrow[k] * scale : 0.f;
  const float v1 = (k + 1 < n && g < n && k + 1 <= g) ? wrow[k + 1] * scale : 0.f;
  uint32_t hi, lo;
  split_f16x2(v0, v1, hi, lo);
  const int q = g / BOUTE_BLKCOLS, c = k / BOUTE_ACHUNK, ncol = plan.ncol[q];
  uint32_t *blk = (uint32_t *)(img + plan.off[q] + (long long)c * 2 * ncol * BOUTE_ACHUNK);
  const int o = sw128_off16(g % BOUTE_BLKCOLS, k % BOUTE_ACHUNK) >> 1;
  const long long base = plan.off[q] + (long long)c * 2 * ncol * BOUTE_ACHUNK;
  (void)base;  // (used by the debug build's checks)
  if (BOUTE_INB(base + 2 * ((ncol * BOUTE_ACHUNK >> 1) + o) + 1, plan.image_halves) &&
      BOUTE_INB(q, plan.nwblk)) {
    blk[o] = hi;
    blk[(ncol * BOUTE_ACHUNK >> 1) + o] = lo;
  }
  return fabsf(v0) < 32768.f && fabsf(v1) < 32768.f;
}

// All of W's image elements, pairs [first, total) by stride (rows of the
// blocks' padded widths, the chunks each block needs).
__device__ __forceinline__ bool pack_elems(const float *W, int ld, const PostPlan &plan,
                                           float scale, uint16_t *img, long long first,
                                           long long stride) {
  const int nblk = plan.nwblk;
  const long long rows = (long long)BOUTE_BLKCOLS * (nblk - 1) + plan.ncol[nblk - 1];
  const int kmax = BOUTE_ACHUNK * plan.kc[nblk - 1];  // pairs per row: kmax / 2
  const long long total = rows * (kmax / 2);
  bool ok = true;
  for (long long e = first; e < total; e += stride) {
    const int g = (int)(e / (kmax / 2)), k = 2 * (int)(e % (kmax / 2));
    if (k / BOUTE_ACHUNK >= plan.kc[g / BOUTE_BLKCOLS]) continue;
    ok &= pack_pair(W + (size_t)(g < plan.npad ? g : 0) * ld, g, k, plan, scale, img);
  }
  return ok;
}

// Error-free product and sum on fp32 pairs (Dekker / Knuth).
__device__ __forceinline__ void two_prod(float a, float b, float &p, float &e) {
  p = a * b;
  e = fmaf(a, b, -p);
}
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
  s = a + b;
  const float bb = s - a;
  e = (a - (s - bb)) + (b - bb);
}

// The standardisation of one outcome column (stride m) by one warp: with
// standardize != 0 the column's mean and 1 / (sample standard deviation) (1
// when that is below 1e-8 or n = 1), as standardize_kernel computes them,
// else 0 and 1; lane 0 stores them.
__device__ __forceinline__ void standardize_stats(const double *y, int n, int m, int standardize,
                                                  int lane, double &mu, double &isd) {
  if (!standardize) {
    if (lane == 0) {
      mu = 0.0;
      isd = 1.0;
    }
    return;
  }
  double sum = 0.0;
  for (int i = lane; i < n; i += 32) sum += y[(size_t)i * m];
  const double mean = warp_sum(sum) / n;
  double ss = 0.0;
  for (int i = lane; i < n; i += 32) {
    const double z = y[(size_t)i * m] - mean;
    ss += z * z;
  }
  ss = warp_sum(ss);
  double sd = n > 1 ? sqrt(ss / (n - 1)) : 1.0;
  if (!(sd >= 1e-8)) sd = 1.0;
  if (lane == 0) {
    mu = mean;
    isd = 1.0 / sd;
  }
}

// The largest preference weight w_j of problem-objective bt (composite
// kernel), by one warp, into its parameter slot.
__device__ __forceinline__ void composite_wmax(float *xt, int bt, const PostPlan &plan, int DP,
                                               int n, int lane) {
  const int cf = xt_chunk_floats(DP);
  float *x0 = xt + (size_t)bt * plan.nxt * cf;
  const float *xw = x0 + BOUTE_KCHUNK * DP;
  float wm = 0.f;
  for (int j = lane; j < n; j += 32) wm = fmaxf(wm, xw[(size_t)(j / BOUTE_KCHUNK) * cf + j % BOUTE_KCHUNK]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
  if (lane == 0) x0[xt_param_offset(DP) + 2 * DP + kParWmax] = wm;
}

// ---- factorisation: one block per (problem, objective) -------------------------
// Blocked right-looking Cholesky of K (its fp32 rounding) in 32-column panels,
// with W = L^-1 formed block row by block row inside the same loop: one warp
// factors and inverts each diagonal block in registers, the panel below is the
// product with that inverse, W_pJ = -W_pp sum_{K=J}^{p-1} L_pK W_KJ, and the
// trailing update uses 4 x 4 register tiles. fp32 arithmetic on the FP32
// pipes: the fp32 factor is as accurate as the posterior needs, while alpha,
// which carries the condition number, gets two steps of iterative refinement
// against the fp64-accurate K = hi + lo with double-float residuals. A pivot
// at or below 16 * eps32 times its original diagonal entry counts as not
// positive. Matrix and inverse live in shared memory (row stride NP+1, NP = n
// rounded up to 32, padded with the identity) when they fit, else in the
// handle's global workspace.
// Threads per block of the two variants: the shared-memory variant runs more
// warps to hide the latency of its short, dependent phases.
template <bool SMEM>
constexpr int fit_threads() { return SMEM ? 512 : 256; }

template <bool SMEM>
__global__ void __launch_bounds__(fit_threads<SMEM>(), 1) fit32_kernel(
    const float *Kh_all, const float *Kl_all, const double *Ys, int standardize, int n, int m,
    float *Aws, float *Wws, float *xt, int DP, int npad, PostPlan plan, uint16_t *bop,
    int kl_smem, int early_trigger, int comp, int *status, const int *fbad, float *Wkeep) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int bad;
  __shared__ uint64_t lbar, lbar_lo;  // K hi; K lo (needed only by the residual)
  __shared__ double ymu, yisd;
  __shared__ __align__(16) float colL[32][64];  // columns of L_pp, zero-padded
  __shared__ float invs[32];                    // 1 / L_cc
  const int bt = blockIdx.x, b = bt / m, t = bt % m;
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5,
            nw = nthr >> 5;
  const int NP = npad, ld = NP + 1;
  const float *Kh = Kh_all + (size_t)bt * n * n, *Kl = Kl_all + (size_t)bt * n * n;
  float *A = SMEM ? sm : Aws + (size_t)bt * NP * ld;
  float *W = SMEM ? sm + (size_t)NP * ld : Wws + (size_t)bt * NP * ld;
  float *vec = SMEM ? sm + 2 * (size_t)NP * ld : sm;  // ylo, dg, y, tv, al, r: 6 x NP
  float *ylo = vec, *dg = vec + NP, *yv = vec + 2 * NP, *tv = vec + 3 * NP, *al = vec + 4 * NP,
        *rv = vec + 5 * NP;
  const double *y = Ys + (size_t)b * n * m + t;
  if (early_trigger) pdl_trigger();  // every block is resident: the posterior may launch
  // standardize != 0: Ys holds raw outcomes; this column is standardised here
  // (zero mean, unit sample standard deviation, as standardize_kernel does)
  if (warp == 0) standardize_stats(y, n, m, standardize, lane, ymu, yisd);  // few fp64 ops
  // everything below reads what the set-up kernel wrote
  pdl_wait();
  // A = K (hi; the lower triangle becomes L, the upper triangle keeps K for the
  // residual), padded with the identity to NP x NP. In shared memory with n
  // even, K hi (and, for n <= 128, K lo) arrive by bulk copy, K hi staged in
  // the W area.
  float *Kls = kl_smem ? vec + 6 * NP : nullptr;  // K lo, n x n (shared)
  const bool bulk = SMEM && (n % 2 == 0);
  if (bulk) {
    if (tid == 0) {
      mbar_init(&lbar, 1);
      mbar_init(&lbar_lo, 1);
      fence_mbar_init();
    }
    __syncthreads();
    if (tid == 0) {
      const uint32_t bytes = (uint32_t)n * n * sizeof(float);
      mbar_arrive_expect_tx(&lbar, bytes);
      bulk_g2s(W, Kh, bytes, &lbar);
      if (kl_smem) {  // lands while the factorisation runs
        mbar_arrive_expect_tx(&lbar_lo, bytes);
        bulk_g2s(Kls, Kl, bytes, &lbar_lo);
      }
    }
  } else if (!fbad) {  // eight independent loads per thread in flight before their stores
    const int nn = n * n;
    for (int base = 0; base < nn; base += 8 * nthr) {
      float v[8], w8[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int e = base + j * nthr + tid;
        v[j] = e < nn ? Kh[e] : 0.f;
        w8[j] = (e < nn && kl_smem) ? Kl[e] : 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int e = base + j * nthr + tid;
        if (e < nn) {
          const int i = e / n, k = e - i * n;
          A[(size_t)i * ld + k] = v[j];
          if (kl_smem) Kls[e] = w8[j];
        }
      }
    }
  }
  for (int e = tid; e < (NP - n) * NP && !fbad; e += nthr) {
    const int i = n + e / NP, k = e % NP;
    if (k <= i) A[(size_t)i * ld + k] = (k == i) ? 1.f : 0.f;
  }
  __syncthreads();
  const double mu_y = ymu, isd_y = yisd;
  if (bulk) {
    if (!mbar_wait(&lbar, 0)) {  // the copy never completed: report, drain, leave
      if (tid == 0) set_status(status, BOUTE_ERR_TIMEOUT);
      mbar_wait(&lbar, 0);
      if (kl_smem) mbar_wait(&lbar_lo, 0);
      return;
    }
    for (int i = warp; i < n; i += nw) {  // a warp per row: no division per entry
      const float *src = W + (size_t)i * n;
      float *dst = A + (size_t)i * ld;
#pragma unroll 4
      for (int k = lane; k < n; k += 32) dst[k] = src[k];
    }
    __syncthreads();
  }
  for (int i = tid; i < NP; i += nthr) {  // standardised y as an fp32 pair
    const double ys = i < n ? (y[(size_t)i * m] - mu_y) * isd_y : 0.0;
    yv[i] = (float)ys;
    ylo[i] = (float)(ys - (double)yv[i]);
    dg[i] = A[(size_t)i * ld + i];
  }
  if (tid == 0) bad = fbad ? fbad[bt] : 0;  // (factored by the blocked kernels)
  for (int e = tid; e < 32 * 64; e += nthr) (&colL[0][0])[e] = 0.f;
  __syncthreads();
  // Operand images of W for the posterior (n <= 160): rows [g_lo, g_hi) of W,
  // warps w0, w0 + nws, ... one row each, lane = pair of columns 2 lane of
  // each 64-wide chunk, scaled by 2^e_W. A block row of W is final once its
  // panel's trailing update is done.
  const float *xpar = xt + (size_t)bt * plan.nxt * xt_chunk_floats(DP) + xt_param_offset(DP) +
                      2 * DP;
  const float wscale = exp2i((int)xpar[kParEW]);
  const int gmax = BOUTE_BLKCOLS * (plan.nwblk - 1) + plan.ncol[plan.nwblk - 1];
  auto pack_rows = [&](int g_lo, int g_hi, int w0, int nws) {
    uint16_t *img = bop + (size_t)bt * plan.image_halves;
    for (int g = g_lo + w0; g < g_hi && g < gmax; g += nws) {
      const float *wr = W + (size_t)g * ld;
      const int kc = plan.kc[g / BOUTE_BLKCOLS];
      for (int c = 0; c < kc; ++c)
        if (!pack_pair(wr, g, BOUTE_ACHUNK * c + 2 * lane, plan, wscale, img))
          set_status(status, BOUTE_ERR_NOT_PD);
    }
  };
  // ---- blocked Cholesky and W = L^-1, 32-column panels -------------------------
  // Iteration p: (a) warp 0 factors the diagonal block, A_pp = L_pp L_pp^T,
  // and warp 1 inverts it one column behind, W_pp = L_pp^-1, both
  // register-resident (lane = row of the block); (b) the panel below, L_rp = A_rp W_pp^T, goes to the still-unused
  // block column p of W, and T_pJ = sum_{K=J}^{p-1} L_pK W_KJ (J < p) is
  // parked, transposed, in the unused upper triangle of W; (c) the trailing
  // update A_ij -= sum_q L_iq L_jq (rows and columns below the panel), the
  // copy of the panel into A, and W_pJ = -W_pp T_pJ. 4 x 4 register tiles (4 x 2
  // for T_pJ and W_pJ).
  const int nb = NP / 32;
  const unsigned FULL = 0xffffffffu;
  for (int p = 0; p < nb && !fbad; ++p) {
    const int p0 = 32 * p;
    if (warp == 0) {
      // Factor. Lane = row of the block. a[] is a window on the lane's row
      // that moves one column right every step (a[0] is always column c), so
      // the step loop runs with static register indices and stays small.
      // Each column of L_pp and 1 / L_cc go to warp 1 through shared memory,
      // one named-barrier handshake per step.
      float a[32];
      float *Ar = A + (size_t)(p0 + lane) * ld + p0;
#pragma unroll
      for (int c = 0; c < 32; ++c) a[c] = (c <= lane) ? Ar[c] : 0.f;
      const float dgl = dg[p0 + lane];
      bool ok = true;
      // steps c0 .. c0 + 7; after step c only a[0 .. 30 - c] still lie in the
      // block, so each quarter of the panel shifts and updates NK entries
      // (the rest are right of the block: never stored, left as they are)
      // The pivot of step c + 1 is lane c + 1's entry after step c, which
      // needs only that lane's own l: it is formed and broadcast before the
      // stores and the row update, whose issue then hides its latency.
      float piv = __shfl_sync(FULL, a[0], 0);
      auto quarter = [&](auto nk, int c0) {
        constexpr int NK = decltype(nk)::value;
#pragma unroll 1
        for (int c = c0; c < c0 + 8; ++c) {
          if (!(piv > 16.f * 1.1920929e-7f * __shfl_sync(FULL, dgl, c))) ok = false;
          float inv = rsqrtf(piv);
          inv = inv * fmaf(-0.5f * piv * inv, inv, 1.5f);  // one Newton step; 1 / L_cc
          const float l = lane > c ? a[0] * inv : (lane == c ? piv * inv : 0.f);
          piv = __shfl_sync(FULL, fmaf(-l, l, a[1]), (c + 1) & 31);  // (unused after c = 31)
          if (lane >= c) Ar[c] = l;
          colL[c][lane] = l;  // colL[c][32..63] stay zero
          if (lane == 0) invs[c] = inv;
          __syncwarp();
          named_barrier_sync(1, 64);  // column c is ready for warp 1
          // trailing update of the lane's row, shifted one column: entries
          // above the lane's diagonal collect values never stored
#pragma unroll
          for (int k = 0; k < NK; ++k) a[k] = fmaf(-l, colL[c][c + 1 + k], a[k + 1]);
        }
      };
      quarter(std::integral_constant<int, 31>{}, 0);
      quarter(std::integral_constant<int, 23>{}, 8);
      quarter(std::integral_constant<int, 15>{}, 16);
      quarter(std::integral_constant<int, 7>{}, 24);
      if (!ok && lane == 0) bad = 1;
    } else if (warp == 1) {
      // Inverse, one column behind the factor. w[] is the lane's row of
      // R = e_lane - sum_{j<c} L_lane,j W_j, which becomes W_pp's row after
      // the division by L_lane,lane. R_c has no entries right of c, so the
      // update at step c touches w[0 .. c] only (NK per quarter of the panel).
      float w[32];
#pragma unroll
      for (int c = 0; c < 32; ++c) w[c] = (c == lane) ? 1.f : 0.f;
      float myinv = 0.f;
      auto quarter = [&](auto nk, int c0) {
        constexpr int NK = decltype(nk)::value;
#pragma unroll 1
        for (int c = c0; c < c0 + 8; ++c) {
          named_barrier_sync(1, 64);  // wait for column c
          const float l = colL[c][lane], inv = invs[c];
          if (lane == c) myinv = inv;
          const float lw = lane > c ? l * inv : 0.f;  // R_i -= (L_ic / L_cc) R_c, rows below c
#pragma unroll
          for (int k = 0; k < NK; ++k) w[k] = fmaf(-lw, __shfl_sync(FULL, w[k], c), w[k]);
        }
      };
      quarter(std::integral_constant<int, 8>{}, 0);
      quarter(std::integral_constant<int, 16>{}, 8);
      quarter(std::integral_constant<int, 24>{}, 16);
      quarter(std::integral_constant<int, 32>{}, 24);
      float *Wr = W + (size_t)(p0 + lane) * ld + p0;
#pragma unroll
      for (int c = 0; c < 32; ++c) Wr[c] = w[c] * myinv;
    } else if (SMEM && p > 0) {
      // the other warps pack the previous block row of W meanwhile
      pack_rows(p0 - 32, p0, warp - 2, nw - 2);
    }
    __syncthreads();
    if (bad) break;
    const int r0 = p0 + 32, rows = NP - r0;
    // (b)
    {
      const int ntr = (rows / 4) * 8, ntt = p * 128;
      for (int tix = tid; tix < ntr + ntt; tix += nthr) {
        float acc[4][4] = {};
        if (tix < ntr) {  // L_rp tile: rows i0.., columns c0.. of the panel
          const int i0 = r0 + 4 * (tix >> 3), c0 = 4 * (tix & 7);
#pragma unroll 4
          for (int q = 0; q < 32; ++q) {
            float x[4], y4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              x[u] = A[(size_t)(i0 + u) * ld + p0 + q];
              y4[u] = W[(size_t)(p0 + c0 + u) * ld + p0 + q];
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(x[u], y4[v], acc[u][v]);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v) W[(size_t)(i0 + u) * ld + p0 + c0 + v] = acc[u][v];
        } else {
          // T_pJ tile of 4 rows x 2 columns (8 x 16 tiles per 32 x 32 block):
          // the sums run over 32 (p - J) terms, so the long ones get twice
          // the threads that 4 x 4 tiles would give them
          const int e = tix - ntr, J = e >> 7, rb = 4 * ((e >> 4) & 7), cb = 2 * (e & 15);
#pragma unroll 4
          for (int q = 32 * J; q < p0; ++q) {
            float x[4], y2[2];
#pragma unroll
            for (int u = 0; u < 4; ++u) x[u] = A[(size_t)(p0 + rb + u) * ld + q];
#pragma unroll
            for (int v = 0; v < 2; ++v) y2[v] = W[(size_t)q * ld + 32 * J + cb + v];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int v = 0; v < 2; ++v) acc[u][v] = fmaf(x[u], y2[v], acc[u][v]);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 2; ++v) W[(size_t)(32 * J + cb + v) * ld + p0 + rb + u] = acc[u][v];
        }
      }
    }
    __syncthreads();
    // (c)
    {
      const int th = rows / 4, ntile = th * (th + 1) / 2, nwt = p * 128;
      for (int tix = tid; tix < ntile + nwt; tix += nthr) {
        float acc[4][4] = {};
        if (tix < ntile) {  // trailing tile (i, j) of the lower triangle
          int ti = (int)((sqrtf(8.f * tix + 1.f) - 1.f) * 0.5f);
          while (ti * (ti + 1) / 2 > tix) --ti;
          while ((ti + 1) * (ti + 2) / 2 <= tix) ++ti;
          const int tj = tix - ti * (ti + 1) / 2;
          const int i0 = r0 + 4 * ti, j0 = r0 + 4 * tj;
#pragma unroll 4
          for (int q = 0; q < 32; ++q) {
            float x[4], y4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              x[u] = W[(size_t)(i0 + u) * ld + p0 + q];
              y4[u] = W[(size_t)(j0 + u) * ld + p0 + q];
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(x[u], y4[v], acc[u][v]);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v)
              if (ti != tj || v <= u) A[(size_t)(i0 + u) * ld + j0 + v] -= acc[u][v];
        } else {  // W_pJ tile = -W_pp T_pJ (W_pp lower, zeros above), 4 rows x 2 columns
          const int e = tix - ntile, J = e >> 7, rb = 4 * ((e >> 4) & 7), cb = 2 * (e & 15);
#pragma unroll 4
          for (int q = 0; q < 32; ++q) {
            float x[4], y2[2];
#pragma unroll
            for (int u = 0; u < 4; ++u) x[u] = W[(size_t)(p0 + rb + u) * ld + p0 + q];
#pragma unroll
            for (int v = 0; v < 2; ++v) y2[v] = W[(size_t)(32 * J + cb + v) * ld + p0 + q];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int v = 0; v < 2; ++v) acc[u][v] = fmaf(x[u], y2[v], acc[u][v]);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 2; ++v) W[(size_t)(p0 + rb + u) * ld + 32 * J + cb + v] = -acc[u][v];
        }
      }
      for (int e = tid; e < rows * 32; e += nthr) {  // the panel into A
        const size_t o = (size_t)(r0 + (e >> 5)) * ld + p0 + (e & 31);
        A[o] = W[o];
      }
    }
    __syncthreads();
  }
  const bool lo_copy = bulk && kl_smem;  // K lo is on its way by bulk copy
  if (bad) {
    if (tid == 0) set_status(status, BOUTE_ERR_NOT_PD);
    if (lo_copy) mbar_wait(&lbar_lo, 0);  // let it land before the block exits
    return;
  }
  // ---- alpha0 = W^T (W y), refined twice against K = hi + lo ---------------------
  // out = W^T (W rhs). Shared-memory variant: the 32 x 32 blocks (I >= J) of
  // W, one warp per block (the diagonal blocks hold zeros above the diagonal,
  // the padding the identity), with the block partial sums in the space of
  // colL (free after the factorisation), added in a fixed order.
  auto solve_blocks = [&](const float *rhs, float *out) {
    float *pw = &colL[0][0], *pt = pw + nb * NP;  // nb x NP each (nb <= 5, NP <= 160)
    const int nblk = nb * (nb + 1) / 2;
    auto block = [&](int e, int &I, int &J) {
      I = 0;
      while ((I + 1) * (I + 2) / 2 <= e) ++I;
      J = e - I * (I + 1) / 2;
    };
    for (int e = warp; e < nblk; e += nw) {  // (W rhs) restricted to block (I, J): lane = row
      int I, J;
      block(e, I, J);
      const float *wr = W + (size_t)(32 * I + lane) * ld + 32 * J;
      const float *x = rhs + 32 * J;
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
      for (int k = 0; k < 32; k += 4) {
        s0 = fmaf(wr[k], x[k], s0);
        s1 = fmaf(wr[k + 1], x[k + 1], s1);
        s2 = fmaf(wr[k + 2], x[k + 2], s2);
        s3 = fmaf(wr[k + 3], x[k + 3], s3);
      }
      pw[J * NP + 32 * I + lane] = (s0 + s1) + (s2 + s3);
    }
    __syncthreads();
    for (int e = warp; e < nblk; e += nw) {  // W^T (W rhs) restricted to block (I, J): lane = column
      int I, J;
      block(e, I, J);
      float v = 0.f;  // (W rhs) of row 32 I + lane
      for (int q = 0; q <= I; ++q) v += pw[q * NP + 32 * I + lane];
      const float *wc = W + (size_t)(32 * I) * ld + 32 * J + lane;
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
      for (int r = 0; r < 32; r += 4) {
        s0 = fmaf(wc[(size_t)r * ld], __shfl_sync(FULL, v, r), s0);
        s1 = fmaf(wc[(size_t)(r + 1) * ld], __shfl_sync(FULL, v, r + 1), s1);
        s2 = fmaf(wc[(size_t)(r + 2) * ld], __shfl_sync(FULL, v, r + 2), s2);
        s3 = fmaf(wc[(size_t)(r + 3) * ld], __shfl_sync(FULL, v, r + 3), s3);
      }
      pt[I * NP + 32 * J + lane] = (s0 + s1) + (s2 + s3);
    }
    __syncthreads();
    for (int k = tid; k < NP; k += nthr) {
      float v = 0.f;
      for (int q = k >> 5; q < nb; ++q) v += pt[q * NP + k];
      out[k] = v;
    }
    __syncthreads();
  };
  // global variant: a warp per row of W (coalesced loads, lanes combined by
  // shuffles in a fixed order), then a thread per column (4 accumulators)
  auto solve = [&](const float *rhs, float *out) {
    if constexpr (SMEM) {
      solve_blocks(rhs, out);
    } else {
    for (int i = warp; i < NP; i += nw) {
      const float *wr = W + (size_t)i * ld;
      float s0 = 0.f, s1 = 0.f;
      int k = lane;
      for (; k + 32 <= i; k += 64) {
        s0 = fmaf(wr[k], rhs[k], s0);
        s1 = fmaf(wr[k + 32], rhs[k + 32], s1);
      }
      if (k <= i) s0 = fmaf(wr[k], rhs[k], s0);
      float v = s0 + s1;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
      if (lane == 0) tv[i] = v;
    }
    __syncthreads();
    for (int k = tid; k < NP; k += nthr) {
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
      int i = k;
      for (; i + 3 < NP; i += 4) {
        s0 = fmaf(W[(size_t)i * ld + k], tv[i], s0);
        s1 = fmaf(W[(size_t)(i + 1) * ld + k], tv[i + 1], s1);
        s2 = fmaf(W[(size_t)(i + 2) * ld + k], tv[i + 2], s2);
        s3 = fmaf(W[(size_t)(i + 3) * ld + k], tv[i + 3], s3);
      }
      for (; i < NP; ++i) s0 = fmaf(W[(size_t)i * ld + k], tv[i], s0);
      out[k] = (s0 + s1) + (s2 + s3);
    }
    __syncthreads();
    }
  };
  solve(yv, al);
  if (lo_copy && !mbar_wait(&lbar_lo, 0)) {  // the copy never completed: report, drain, leave
    if (tid == 0) set_status(status, BOUTE_ERR_TIMEOUT);
    mbar_wait(&lbar_lo, 0);
    return;
  }
  auto residual = [&]() {
    // residual r = y - K alpha in double-float. Shared-memory variant: one
    // warp per 32 x 32 block (I, J) of K, lane = row, two independent chains per
    // lane; K lo through its symmetry (K lo[k][i], conflict-free across the
    // lanes), from shared memory when it fits there; K hi from the upper
    // triangle of A: at (k, i) below the diagonal blocks, at (i, k) above them,
    // each with one fixed load form (a per-entry choice of address costs more
    // than the arithmetic), and in the diagonal blocks both loaded and the
    // value selected, the diagonal from dg. Indices past n are clamped and
    // alpha is zero there (padding), so those terms add exact zeros. The block
    // partial sums (hi, lo) go to the space of colL and are added per row in a
    // fixed order.
    if (SMEM) {
      float *ph = &colL[0][0], *pl = ph + nb * NP;  // nb x NP each
      const float *Klsm = vec + 6 * NP;  // = Kls when kl_smem (shared-space pointer)
      for (int e = warp; e < nb * nb; e += nw) {
        const int I = e / nb, J = e - I * nb, ci = min(32 * I + lane, n - 1);
        const float *alJ = al + 32 * J;
        float sh[2] = {0.f, 0.f}, sl[2] = {0.f, 0.f};
        auto run = [&](auto form, auto lo_smem) {
          constexpr int F = decltype(form)::value;  // 0: below, 1: above, 2: diagonal block
          constexpr bool LS = decltype(lo_smem)::value;
          const float di = dg[ci];
  #pragma unroll 8
          for (int kk = 0; kk < 32; ++kk) {
            const int kc = min(32 * J + kk, n - 1);
            float h;
            if (F == 0) {
              h = A[kc * ld + ci];
            } else if (F == 1) {
              h = A[ci * ld + kc];
            } else {
              const float x = A[kc * ld + ci], y = A[ci * ld + kc];
              h = kc < ci ? x : y;
              h = kc == ci ? di : h;
            }
            const float l = LS ? Klsm[kc * n + ci] : Kl[(size_t)kc * n + ci];
            const float a = alJ[kk];  // zero from n on
            float pr, er, s_, e2;
            two_prod(h, a, pr, er);
            two_sum(sh[kk & 1], pr, s_, e2);
            sh[kk & 1] = s_;
            sl[kk & 1] += e2 + fmaf(l, a, er);
          }
        };
        auto pick = [&](auto lo_smem) {
          if (I > J) run(std::integral_constant<int, 0>{}, lo_smem);
          else if (I < J) run(std::integral_constant<int, 1>{}, lo_smem);
          else run(std::integral_constant<int, 2>{}, lo_smem);
        };
        if (kl_smem) pick(std::true_type{});
        else pick(std::false_type{});
        float s_, e2;
        two_sum(sh[0], sh[1], s_, e2);
        ph[J * NP + 32 * I + lane] = s_;
        pl[J * NP + 32 * I + lane] = (sl[0] + sl[1]) + e2;
      }
      __syncthreads();
      for (int i = tid; i < NP; i += nthr) {
        float sh = 0.f, sl = 0.f;
        for (int J = 0; J < nb; ++J) {
          float s_, e2;
          two_sum(sh, ph[J * NP + i], s_, e2);
          sh = s_;
          sl += pl[J * NP + i] + e2;
        }
        if (i < n) rv[i] = (yv[i] - sh) + (ylo[i] - sl);
      }
    } else {
      // global variant: two rows per half warp at a time, all their loads
      // issued before the arithmetic
      const int half = lane >> 4, hl = lane & 15;
      for (int i0 = 2 * warp + half; i0 < NP; i0 += 4 * nw) {
        const int rows[2] = {i0, i0 + 2 * nw};
        float sh[2] = {0.f, 0.f}, sl[2] = {0.f, 0.f};
        for (int k0 = 0; k0 < n; k0 += 128) {
          float h8[2][8], l8[2][8], a8[8];
  #pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int k = k0 + hl + 16 * u;
            a8[u] = k < n ? al[k] : 0.f;
  #pragma unroll
            for (int q = 0; q < 2; ++q) {
              const bool ok = k < n && rows[q] < n;
              h8[q][u] = ok ? Kh[(size_t)rows[q] * n + k] : 0.f;
              l8[q][u] = ok ? Kl[(size_t)rows[q] * n + k] : 0.f;
            }
          }
  #pragma unroll
          for (int q = 0; q < 2; ++q)
  #pragma unroll
            for (int u = 0; u < 8; ++u) {
              float pr, e, s_, e2;
              two_prod(h8[q][u], a8[u], pr, e);
              two_sum(sh[q], pr, s_, e2);
              sh[q] = s_;
              sl[q] += e2 + fmaf(l8[q][u], a8[u], e);
            }
        }
  #pragma unroll
        for (int q = 0; q < 2; ++q) {
  #pragma unroll
          for (int o = 8; o > 0; o >>= 1) {  // within the half warp
            const float oh = __shfl_xor_sync(FULL, sh[q], o);
            const float ol = __shfl_xor_sync(FULL, sl[q], o);
            float s_, e;
            two_sum(sh[q], oh, s_, e);
            sh[q] = s_;
            sl[q] += ol + e;
          }
          if (hl == 0 && rows[q] < n) rv[rows[q]] = (yv[rows[q]] - sh[q]) + (ylo[rows[q]] - sl[q]);
        }
      }
    }
  };
  // two refinement steps: alpha carries the condition number of K, and the
  // posterior mean amplifies its error by sum_j |K*_j alpha_j| / |mean|
  // The second correction is kept exactly: alpha = hi + lo, hi = fl(alpha +
  // delta), lo its rounding error (in rv), for the posterior's fp64 path.
  for (int step = 0; step < 2; ++step) {
    residual();
    for (int i = n + tid; i < NP; i += nthr) rv[i] = 0.f;
    __syncthreads();
    solve(rv, rv);
    for (int k = tid; k < NP; k += nthr) {
      if (step == 0) {
        al[k] += rv[k];
      } else {
        float s_, e;
        two_sum(al[k], rv[k], s_, e);
        al[k] = s_;
        rv[k] = e;
      }
    }
    __syncthreads();
  }
  // outputs: the operand images of W (packed here from shared memory; the
  // global variant leaves W in the workspace for pack_kernel), alpha into the
  // side input
  if (SMEM) pack_rows(NP - 32, NP, warp, nw);  // the last block row (the others: above)
  if (SMEM && Wkeep) {  // W in global memory too (the in-sample preparation, the
                        // acquisition's gradient), its lower triangle
    float *dst = Wkeep + (size_t)bt * NP * ld;
    for (int i = warp; i < n; i += nw)
      for (int k = lane; k <= i; k += 32) dst[(size_t)i * ld + k] = W[(size_t)i * ld + k];
  }
  const int cf = xt_chunk_floats(DP);
  float *xa = xt + (size_t)bt * plan.nxt * cf + xt_alpha_offset(DP);
  for (int k = tid; k < BOUTE_KCHUNK * plan.nxt; k += nthr) {
    float *q = xa + (size_t)(k / BOUTE_KCHUNK) * cf + k % BOUTE_KCHUNK;
    q[0] = k < n ? al[k] : 0.f;
    q[BOUTE_KCHUNK] = k < n ? rv[k] : 0.f;
  }
  if (comp && warp == nw - 1) composite_wmax(xt, bt, plan, DP, n, lane);
}

// ---- the global-workspace factorisation across many blocks -------------------------
// For n > 160 the three phases of every 32-column panel of fit32_kernel's loop
// run as three kernels, each over as many blocks as its tiles fill (a grid of
// x blocks per problem-objective y), with programmatic dependent launch in
// between: (a) fitb_diag_kernel factors and inverts the diagonal block, (b)
// fitb_panel_kernel forms the panel below and the partial sums of T_pJ, (c)
// fitb_update_kernel applies the trailing update, adds the partials in a fixed
// order (the result does not depend on the grid), forms W's block row and
// copies the panel into A. The tiles' arithmetic is the same as in the
// one-block loop; the fitr_* kernels then form alpha from the factored
// workspace. A non-positive pivot marks the problem-objective in fbad
// and its later kernels return at once.
constexpr int kFitbThreads = 256;

// A = K hi below the diagonal, the identity on the padding; fbad cleared.
__global__ void __launch_bounds__(kFitbThreads) fitb_load_kernel(const float *Kh_all, int n,
                                                                 int NP, float *Aws, int *fbad) {
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.y, ld = NP + 1;
  const float *Kh = Kh_all + (size_t)bt * n * n;
  float *A = Aws + (size_t)bt * NP * ld;
  const long long tot = (long long)NP * NP;
  for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < tot;
       e += (long long)gridDim.x * blockDim.x) {
    const int i = (int)(e / NP), k = (int)(e % NP);
    if (k > i) continue;
    A[(size_t)i * ld + k] = i < n ? Kh[(size_t)i * n + k] : (k == i ? 1.f : 0.f);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) fbad[bt] = 0;
}

// (a) one block of two warps per problem-objective: warp 0 factors A_pp in
// registers (the pivot test against K's own diagonal), warp 1 inverts it one
// column behind into W_pp, as in fit32_kernel.
__global__ void __launch_bounds__(64) fitb_diag_kernel(const float *Kh_all, int n, int NP,
                                                       float *Aws, float *Wws, int p,
                                                       int *fbad) {
  __shared__ __align__(16) float colL[32][64];
  __shared__ float invs[32];
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.x, ld = NP + 1, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (fbad[bt]) return;
  const float *Kh = Kh_all + (size_t)bt * n * n;
  float *A = Aws + (size_t)bt * NP * ld, *W = Wws + (size_t)bt * NP * ld;
  const int p0 = 32 * p;
  const unsigned FULL = 0xffffffffu;
  for (int e = threadIdx.x; e < 32 * 64; e += 64) (&colL[0][0])[e] = 0.f;
  __syncthreads();
  if (warp == 0) {
    float a[32];
    float *Ar = A + (size_t)(p0 + lane) * ld + p0;
#pragma unroll
    for (int c = 0; c < 32; ++c) a[c] = (c <= lane) ? Ar[c] : 0.f;
    const int gi = p0 + lane;
    const float dgl = gi < n ? Kh[(size_t)gi * n + gi] : 1.f;
    bool ok = true;
    float piv = __shfl_sync(FULL, a[0], 0);
    auto quarter = [&](auto nk, int c0) {
      constexpr int NK = decltype(nk)::value;
#pragma unroll 1
      for (int c = c0; c < c0 + 8; ++c) {
        if (!(piv > 16.f * 1.1920929e-7f * __shfl_sync(FULL, dgl, c))) ok = false;
        float inv = rsqrtf(piv);
        inv = inv * fmaf(-0.5f * piv * inv, inv, 1.5f);  // one Newton step; 1 / L_cc
        const float l = lane > c ? a[0] * inv : (lane == c ? piv * inv : 0.f);
        piv = __shfl_sync(FULL, fmaf(-l, l, a[1]), (c + 1) & 31);
        if (lane >= c) Ar[c] = l;
        colL[c][lane] = l;
        if (lane == 0) invs[c] = inv;
        __syncwarp();
        named_barrier_sync(1, 64);  // column c is ready for warp 1
#pragma unroll
        for (int k = 0; k < NK; ++k) a[k] = fmaf(-l, colL[c][c + 1 + k], a[k + 1]);
      }
    };
    quarter(std::integral_constant<int, 31>{}, 0);
    quarter(std::integral_constant<int, 23>{}, 8);
    quarter(std::integral_constant<int, 15>{}, 16);
    quarter(std::integral_constant<int, 7>{}, 24);
    if (__any_sync(FULL, !ok) && lane == 0) fbad[bt] = 1;
  } else {
    float w[32];
#pragma unroll
    for (int c = 0; c < 32; ++c) w[c] = (c == lane) ? 1.f : 0.f;
    float myinv = 0.f;
    auto quarter = [&](auto nk, int c0) {
      constexpr int NK = decltype(nk)::value;
#pragma unroll 1
      for (int c = c0; c < c0 + 8; ++c) {
        named_barrier_sync(1, 64);  // wait for column c
        const float l = colL[c][lane], inv = invs[c];
        if (lane == c) myinv = inv;
        const float lw = lane > c ? l * inv : 0.f;
#pragma unroll
        for (int k = 0; k < NK; ++k) w[k] = fmaf(-lw, __shfl_sync(FULL, w[k], c), w[k]);
      }
    };
    quarter(std::integral_constant<int, 8>{}, 0);
    quarter(std::integral_constant<int, 16>{}, 8);
    quarter(std::integral_constant<int, 24>{}, 16);
    quarter(std::integral_constant<int, 32>{}, 24);
    float *Wr = W + (size_t)(p0 + lane) * ld + p0;
#pragma unroll
    for (int c = 0; c < 32; ++c) Wr[c] = w[c] * myinv;
  }
}

// The 32 x 32 tiles of (b) and (c): a block of kFitbThreads threads stages
// its two operand tiles in shared memory (row stride 33) with coalesced loads
// and forms a 2 x 2 output tile per thread (rows rb, rb + 1, columns cb,
// cb + 1), each output an fmaf chain over q = 0..31 in order.
using Tile = float[32][33];

__device__ __forceinline__ void fitb_tile_load(Tile &dst, const float *src, int ld, int tid) {
#pragma unroll
  for (int j = 0; j < 1024 / kFitbThreads; ++j) {
    const int x = tid + kFitbThreads * j, r = x >> 5, c = x & 31;
    dst[r][c] = src[(size_t)r * ld + c];
  }
}

// acc[u][v] += sum_q X[rb + u][q] Y[cb + v][q]  (X Y^T)
__device__ __forceinline__ void fitb_mma_abt(const Tile &X, const Tile &Y, int rb, int cb,
                                             float (&acc)[2][2]) {
#pragma unroll 8
  for (int q = 0; q < 32; ++q) {
    const float x0 = X[rb][q], x1 = X[rb + 1][q], y0 = Y[cb][q], y1 = Y[cb + 1][q];
    acc[0][0] = fmaf(x0, y0, acc[0][0]);
    acc[0][1] = fmaf(x0, y1, acc[0][1]);
    acc[1][0] = fmaf(x1, y0, acc[1][0]);
    acc[1][1] = fmaf(x1, y1, acc[1][1]);
  }
}

// acc[u][v] += sum_q X[rb + u][q] Y[q][cb + v]  (X Y)
__device__ __forceinline__ void fitb_mma_ab(const Tile &X, const Tile &Y, int rb, int cb,
                                            float (&acc)[2][2]) {
#pragma unroll 8
  for (int q = 0; q < 32; ++q) {
    const float x0 = X[rb][q], x1 = X[rb + 1][q], y0 = Y[q][cb], y1 = Y[q][cb + 1];
    acc[0][0] = fmaf(x0, y0, acc[0][0]);
    acc[0][1] = fmaf(x0, y1, acc[0][1]);
    acc[1][0] = fmaf(x1, y0, acc[1][0]);
    acc[1][1] = fmaf(x1, y1, acc[1][1]);
  }
}

// (b) the panel, L_Rp = A_Rp W_pp^T, in place in A for every block row R > p
// (one work item each), and the partial sums of T_pJ = sum_{K=J}^{p-1} L_pK
// W_KJ (J < p) into the workspace tpart: T_pJ's K range is split into chunks
// of kFitbChunk blocks, one work item each, so that no item runs more than
// kFitbChunk tile steps and the panel's critical path stays short for every p.
// tpart holds, per problem-objective, nbw x ncw tiles of 32 x 32 floats (J,
// chunk), nbw = NP / 32 and ncw = ceil(nbw / kFitbChunk).
constexpr int kFitbChunk = 4;
__host__ __device__ __forceinline__ int fitb_t_items(int p) {
  int t = 0;
  for (int J = 0; J < p; ++J) t += (p - J + kFitbChunk - 1) / kFitbChunk;
  return t;
}

__global__ void __launch_bounds__(kFitbThreads) fitb_panel_kernel(int NP, float *Aws,
                                                                  const float *Wws, int p,
                                                                  const int *fbad, float *tpart) {
  __shared__ Tile Xs, Ys;
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.y, ld = NP + 1, tid = threadIdx.x;
  if (fbad[bt]) return;
  float *A = Aws + (size_t)bt * NP * ld;
  const float *W = Wws + (size_t)bt * NP * ld;
  const int nbw = NP / 32, ncw = (nbw + kFitbChunk - 1) / kFitbChunk, p0 = 32 * p;
  const int nr = nbw - 1 - p, items = nr + fitb_t_items(p);
  const int rb = 2 * (tid >> 4), cb = 2 * (tid & 15);
  bool wpp = false;  // W_pp staged in Ys
  for (int item = blockIdx.x; item < items; item += gridDim.x) {
    float acc[2][2] = {};
    if (item < nr) {  // L_Rp = A_Rp W_pp^T
      float *ar = A + (size_t)(p0 + 32 + 32 * item) * ld + p0;
      __syncthreads();  // the previous item's tiles are consumed
      fitb_tile_load(Xs, ar, ld, tid);
      if (!wpp) fitb_tile_load(Ys, W + (size_t)p0 * ld + p0, ld, tid);
      wpp = true;
      __syncthreads();
      fitb_mma_abt(Xs, Ys, rb, cb, acc);
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int v = 0; v < 2; ++v) ar[(size_t)(rb + u) * ld + cb + v] = acc[u][v];
      continue;
    }
    // the item's (J, c): K in [J + c kFitbChunk, min(J + (c + 1) kFitbChunk, p))
    int J = 0, rest = item - nr;
    while (rest >= (p - J + kFitbChunk - 1) / kFitbChunk) {
      rest -= (p - J + kFitbChunk - 1) / kFitbChunk;
      ++J;
    }
    const int c = rest, Kb = J + c * kFitbChunk, Ke = min(Kb + kFitbChunk, p);
    wpp = false;
    for (int K = Kb; K < Ke; ++K) {
      __syncthreads();
      fitb_tile_load(Xs, A + (size_t)p0 * ld + 32 * K, ld, tid);
      fitb_tile_load(Ys, W + (size_t)(32 * K) * ld + 32 * J, ld, tid);
      __syncthreads();
      fitb_mma_ab(Xs, Ys, rb, cb, acc);
    }
    const size_t tile = ((size_t)bt * nbw + J) * ncw + c;
    if (!BOUTE_INB(tile, (size_t)gridDim.y * nbw * ncw)) continue;
    float *tp = tpart + tile * 1024;
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int v = 0; v < 2; ++v) tp[(rb + u) * 32 + cb + v] = acc[u][v];
  }
}

// (c) W_pJ = -W_pp T_pJ for J < p (one work item each; T_pJ the partials
// added in chunk order, so the result does not depend on the grid), then the
// trailing update A_IJ -= L_Ip L_Jp^T for p < J <= I (one item per 32 x 32
// tile; the lower triangle of the diagonal tiles).
__global__ void __launch_bounds__(kFitbThreads) fitb_update_kernel(int NP, float *Aws,
                                                                   float *Wws, int p,
                                                                   const int *fbad,
                                                                   const float *tpart) {
  __shared__ Tile Xs, Ys;
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.y, ld = NP + 1, tid = threadIdx.x;
  if (fbad[bt]) return;
  float *A = Aws + (size_t)bt * NP * ld;
  float *W = Wws + (size_t)bt * NP * ld;
  const int nbw = NP / 32, ncw = (nbw + kFitbChunk - 1) / kFitbChunk, p0 = 32 * p;
  const int T = nbw - 1 - p, items = p + T * (T + 1) / 2;
  const int rb = 2 * (tid >> 4), cb = 2 * (tid & 15);
  bool wpp = false;  // W_pp staged in Xs
  for (int item = blockIdx.x; item < items; item += gridDim.x) {
    float acc[2][2] = {};
    if (item < p) {  // W_pJ, J = item
      const int J = item, nc = (p - J + kFitbChunk - 1) / kFitbChunk;
      const float *tp = tpart + ((size_t)bt * nbw + J) * ncw * 1024;
      __syncthreads();
      if (!wpp) fitb_tile_load(Xs, W + (size_t)p0 * ld + p0, ld, tid);
      wpp = true;
#pragma unroll
      for (int j = 0; j < 1024 / kFitbThreads; ++j) {
        const int x = tid + kFitbThreads * j;
        float t = 0.f;
        for (int c = 0; c < nc; ++c) t += tp[(size_t)c * 1024 + x];
        Ys[x >> 5][x & 31] = t;
      }
      __syncthreads();
      fitb_mma_ab(Xs, Ys, rb, cb, acc);
      float *wr = W + (size_t)p0 * ld + 32 * J;
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int v = 0; v < 2; ++v) wr[(size_t)(rb + u) * ld + cb + v] = -acc[u][v];
      continue;
    }
    const int e = item - p;
    int ti = (int)((sqrtf(8.f * e + 1.f) - 1.f) * 0.5f);
    while (ti * (ti + 1) / 2 > e) --ti;
    while ((ti + 1) * (ti + 2) / 2 <= e) ++ti;
    const int tj = e - ti * (ti + 1) / 2, I = p + 1 + ti, J = p + 1 + tj;
    wpp = false;
    __syncthreads();
    fitb_tile_load(Xs, A + (size_t)(32 * I) * ld + p0, ld, tid);
    fitb_tile_load(Ys, A + (size_t)(32 * J) * ld + p0, ld, tid);
    __syncthreads();
    fitb_mma_abt(Xs, Ys, rb, cb, acc);
    float *ar = A + (size_t)(32 * I) * ld + 32 * J;
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int v = 0; v < 2; ++v)
        if (I != J || cb + v <= rb + u) ar[(size_t)(rb + u) * ld + cb + v] -= acc[u][v];
  }
}

// ---- alpha on the blocked path, across many blocks -----------------------------
// After the blocked factorisation, fit32_kernel's alpha (alpha0 = W^T (W y),
// then two refinement steps against K = hi + lo with double-float residuals,
// the second correction kept as alpha's lo part) runs as a chain of kernels,
// each spread over many blocks per problem-objective (a grid of x blocks per
// problem-objective y): fitr_init_kernel (the standardised y, the output
// padding), then per solve fitr_wx_kernel (t = W rhs, a warp per row) and
// fitr_wtx_kernel (W^T t, 32 columns per block, the rows split over its warps
// and added in a fixed order), and fitr_resid_kernel (r = y - K alpha, a half
// warp per row) between the solves. The vectors live in the workspace fvec,
// kFitrVecs x NP floats per problem-objective.
enum { kVy = 0, kVylo = 1, kVal = 2, kVlo = 3, kVt = 4, kVr = 5, kFitrVecs = 6 };

__global__ void __launch_bounds__(256) fitr_init_kernel(const double *Ys, int standardize, int n,
                                                        int m, int NP, float *fvec, float *xt,
                                                        int DP, PostPlan plan, int comp,
                                                        int *status, const int *fbad) {
  __shared__ double ymu, yisd;
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.x, b = bt / m, t = bt % m, tid = threadIdx.x, lane = tid & 31;
  if (fbad[bt]) {
    if (tid == 0) set_status(status, BOUTE_ERR_NOT_PD);
    return;
  }
  const double *y = Ys + (size_t)b * n * m + t;
  if (tid < 32) standardize_stats(y, n, m, standardize, lane, ymu, yisd);
  __syncthreads();
  float *v = fvec + (size_t)bt * kFitrVecs * NP;
  for (int i = tid; i < NP; i += blockDim.x) {  // standardised y as an fp32 pair
    const double ys = i < n ? (y[(size_t)i * m] - ymu) * yisd : 0.0;
    const float hi = (float)ys;
    v[kVy * NP + i] = hi;
    v[kVylo * NP + i] = (float)(ys - (double)hi);
  }
  const int cf = xt_chunk_floats(DP);
  float *xa = xt + (size_t)bt * plan.nxt * cf + xt_alpha_offset(DP);
  for (int k = n + tid; k < BOUTE_KCHUNK * plan.nxt; k += blockDim.x) {  // alpha's padding
    float *q = xa + (size_t)(k / BOUTE_KCHUNK) * cf + k % BOUTE_KCHUNK;
    q[0] = 0.f;
    q[BOUTE_KCHUNK] = 0.f;
  }
  if (comp && tid < 32) composite_wmax(xt, bt, plan, DP, n, lane);
}

// t = W rhs (W lower triangular): a warp per row, two accumulators per lane,
// the lanes combined by shuffles in a fixed order.
__global__ void __launch_bounds__(256) fitr_wx_kernel(int NP, const float *Wws, float *fvec,
                                                      int src, const int *fbad) {
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.y, ld = NP + 1, lane = threadIdx.x & 31;
  if (fbad[bt]) return;
  const float *W = Wws + (size_t)bt * NP * ld;
  float *v = fvec + (size_t)bt * kFitrVecs * NP;
  const float *rhs = v + src * NP;
  const int i = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (i >= NP) return;
  const float *wr = W + (size_t)i * ld;
  float s0 = 0.f, s1 = 0.f;
  int k = lane;
  for (; k + 32 <= i; k += 64) {
    s0 = fmaf(wr[k], rhs[k], s0);
    s1 = fmaf(wr[k + 32], rhs[k + 32], s1);
  }
  if (k <= i) s0 = fmaf(wr[k], rhs[k], s0);
  float r = s0 + s1;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
  if (lane == 0 && BOUTE_INB(i, NP)) v[kVt * NP + i] = r;
}

// W^T t for columns [32 x, 32 x + 32): lane = column, warp w takes the rows
// i = k0 + w, k0 + w + 8, ... (those at or below the column's diagonal), the
// eight partial sums added in a fixed order. mode 0: alpha = the result;
// mode 1: alpha += the result; mode 2: alpha + the result kept exactly as a
// pair (hi, lo), written with alpha's padding into the side input.
__global__ void __launch_bounds__(256) fitr_wtx_kernel(int NP, int n, const float *Wws,
                                                       float *fvec, int mode, float *xt, int DP,
                                                       PostPlan plan, const int *fbad) {
  __shared__ float part[8][33];
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.y, ld = NP + 1, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (fbad[bt]) return;
  const float *W = Wws + (size_t)bt * NP * ld;
  float *v = fvec + (size_t)bt * kFitrVecs * NP;
  const float *tv = v + kVt * NP;
  const int k0 = 32 * blockIdx.x, k = k0 + lane;
  float s0 = 0.f, s1 = 0.f;  // entries above the diagonal are never loaded
  int i = k0 + warp;
  for (; i + 8 < NP; i += 16) {
    const float w0 = i >= k ? W[(size_t)i * ld + k] : 0.f;
    const float w1 = i + 8 >= k ? W[(size_t)(i + 8) * ld + k] : 0.f;
    s0 = fmaf(w0, tv[i], s0);
    s1 = fmaf(w1, tv[i + 8], s1);
  }
  if (i < NP && i >= k) s0 = fmaf(W[(size_t)i * ld + k], tv[i], s0);
  part[warp][lane] = s0 + s1;
  __syncthreads();
  if (warp == 0 && BOUTE_INB(k, NP)) {
    const float out = ((part[0][lane] + part[1][lane]) + (part[2][lane] + part[3][lane])) +
                      ((part[4][lane] + part[5][lane]) + (part[6][lane] + part[7][lane]));
    float *al = v + kVal * NP;
    if (mode == 0) {
      al[k] = out;
    } else if (mode == 1) {
      al[k] += out;
    } else {
      float hi, lo;
      two_sum(al[k], out, hi, lo);
      al[k] = hi;
      v[kVlo * NP + k] = lo;
      if (k < n) {
        const int cf = xt_chunk_floats(DP);
        float *q = xt + (size_t)bt * plan.nxt * cf + xt_alpha_offset(DP) +
                   (size_t)(k / BOUTE_KCHUNK) * cf + k % BOUTE_KCHUNK;
        q[0] = hi;
        q[BOUTE_KCHUNK] = lo;
      }
    }
  }
}

// r = y - K alpha in double-float (K = hi + lo, alpha zero from n on): a half
// warp per row, eight loads of each of K hi and K lo per lane in flight, the
// lanes combined by shuffles in a fixed order; zero from n on.
__global__ void __launch_bounds__(256) fitr_resid_kernel(const float *Kh_all, const float *Kl_all,
                                                         int n, int NP, float *fvec,
                                                         const int *fbad) {
  pdl_wait();
  pdl_trigger();
  const int bt = blockIdx.y, lane = threadIdx.x & 31, hl = lane & 15;
  if (fbad[bt]) return;
  const float *Kh = Kh_all + (size_t)bt * n * n, *Kl = Kl_all + (size_t)bt * n * n;
  float *v = fvec + (size_t)bt * kFitrVecs * NP;
  const float *al = v + kVal * NP;
  const int i = blockIdx.x * 16 + (threadIdx.x >> 4);
  if (i >= NP) return;  // a whole half warp
  float sh = 0.f, sl = 0.f;
  if (i < n) {
    for (int k0 = 0; k0 < n; k0 += 128) {
      float h8[8], l8[8], a8[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int k = k0 + hl + 16 * u;
        const bool ok = k < n;
        a8[u] = ok ? al[k] : 0.f;
        h8[u] = ok ? Kh[(size_t)i * n + k] : 0.f;
        l8[u] = ok ? Kl[(size_t)i * n + k] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        float pr, e, s_, e2;
        two_prod(h8[u], a8[u], pr, e);
        two_sum(sh, pr, s_, e2);
        sh = s_;
        sl += e2 + fmaf(l8[u], a8[u], e);
      }
    }
  }
  const unsigned half = 0xffffu << (lane & 16);
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) {  // within the half warp
    const float oh = __shfl_xor_sync(half, sh, o);
    const float ol = __shfl_xor_sync(half, sl, o);
    float s_, e;
    two_sum(sh, oh, s_, e);
    sh = s_;
    sl += ol + e;
  }
  if (hl == 0 && BOUTE_INB(i, NP))
    v[kVr * NP + i] = i < n ? (v[kVy * NP + i] - sh) + (v[kVylo * NP + i] - sl) : 0.f;
}

// ---- operand images of L^-1 as fp16 hi/lo, swizzled (global-workspace fit) ----
__global__ void pack_kernel(const float *Wws, PostPlan plan, uint16_t *bop, const float *xt,
                            int DP, int *status) {
  if (*status == BOUTE_ERR_NOT_PD) return;
  const size_t bt = blockIdx.y;
  const int ld = plan.npad + 1;
  const float *xpar = xt + bt * plan.nxt * xt_chunk_floats(DP) + xt_param_offset(DP) + 2 * DP;
  if (!pack_elems(Wws + bt * plan.npad * ld, ld, plan, exp2i((int)xpar[kParEW]),
                  bop + bt * plan.image_halves,
                  (long long)blockIdx.x * blockDim.x + threadIdx.x,
                  (long long)gridDim.x * blockDim.x))
    set_status(status, BOUTE_ERR_NOT_PD);
}

}  // namespace

// Outcome transforms alone (codes != 0), elementwise: Yt = t(Y), count
// values of m objectives.
__global__ void transform_kernel(const double *Y, long long count, int m, int codes, double *Yt) {
  for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < count;
       e += (long long)gridDim.x * blockDim.x)
    Yt[e] = outcome_transform(Y[e], objective_code(codes, (int)(e % m)));
}

int launch_outcome_transform(const double *Y, long long count, int m, int codes, double *Yt,
                             cudaStream_t s) {
  const int blocks = (int)std::min<long long>((count + 255) / 256, 1024);
  transform_kernel<<<std::max(blocks, 1), 256, 0, s>>>(Y, count, m, codes, Yt);
  count_launch();
  return last_launch_status();
}

int launch_standardize(const double *Y, int B, int n, int m, int codes, double *Ys,
                       cudaStream_t s) {
  standardize_kernel<<<B * m, 256, 0, s>>>(Y, n, m, codes, Ys);
  count_launch();
  return last_launch_status();
}

// The shared-memory variant holds n up to 160 (n rounded up to 32).
bool fit_uses_smem(int npad) { return npad <= 160; }

size_t fit_tpart_floats(int npad, int BM) {
  if (fit_uses_smem(npad) || 4 * BM > num_sms()) return 0;  // no blocked factorisation
  const int nbw = npad / 32, ncw = (nbw + kFitbChunk - 1) / kFitbChunk;
  return (size_t)BM * nbw * ncw * 1024;
}

size_t fit_fvec_floats(int npad, int BM) {
  return fit_tpart_floats(npad, BM) ? (size_t)BM * kFitrVecs * npad : 0;
}

// Dynamic shared memory of the shared-memory fit: A and W (np x (np+1)), six
// vectors, and K lo (n x n) when n <= 128.
static bool fit_kl_in_smem(int n) { return n <= 128; }
size_t fit_smem_bytes(int np, int n) {
  return (2 * (size_t)np * (np + 1) + 6 * (size_t)np + (fit_kl_in_smem(n) ? (size_t)n * n : 0)) *
         sizeof(float);
}

// Ys: standardised outcomes, or raw outcomes when standardize != 0.
static int launch_fit_impl(Gp *gp, const double *X, const double *Ys, int standardize,
                           const double *ls, const double *s2, const double *noise,
                           cudaStream_t s, cudaEvent_t setup_done = nullptr) {
  const int n = gp->n, d = gp->d, m = gp->m, BM = gp->B * gp->m;
  const int npad = gp->plan.npad, xpad = BOUTE_KCHUNK * gp->plan.nxt;
  const int nkt = kmat_units(n);
  const int sms = num_sms();
  // side-input blocks: as many as leave one block per SM (K blocks first), 2 .. 16
  const int nprep = std::max(2, std::min(16, sms / BM - nkt));
  // early triggers only when every block of the grid is resident at once (8
  // set-up blocks per SM beside the fit's blocks; one fit block per SM), so
  // that waiting successors can never hold resources a later block needs
  const long long setup_blocks = (long long)(nkt + nprep) * BM;
  const int setup_early = setup_blocks <= 8LL * (sms - BM) ? 1 : 0;
  const int fit_early = 2 * BM <= sms ? 1 : 0;
  auto setup = [&](auto kern) {
    prefer_shared(kern);
    kern<<<dim3(nkt + nprep, BM), kSetupThreads, 0, s>>>(X, n, d, m, gp->DP, xpad, ls, s2, noise,
                                                         gp->Kh, gp->Kl, gp->xt, gp->s2f, nkt,
                                                         nprep, setup_early, gp->status,
                                                         gp->kpar, gp->dtau);
  };
  if (gp->kern) setup(fit_setup_kernel<true>);
  else setup(fit_setup_kernel<false>);
  if (setup_done && cudaEventRecord(setup_done, s) != cudaSuccess) return last_launch_status();
  // the one-block fits already fill the GPU when there are many problem-
  // objectives; with few, the blocked factorisation spreads each over blocks
  const bool blocked = !fit_uses_smem(npad) && 4 * BM <= sms && gp->tpart && gp->fvec;
  if (fit_uses_smem(npad) || !blocked) {
    const bool sm_fit = fit_uses_smem(npad);
    if (sm_fit) {
      const size_t smem = fit_smem_bytes(npad, n);
      prefer_shared(fit32_kernel<true>);
      cudaFuncSetAttribute(fit32_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
      launch_pdl(fit32_kernel<true>, dim3(BM), dim3(fit_threads<true>()), smem, s, gp->Kh,
                 gp->Kl, Ys, standardize, n, m, gp->Aws, gp->Wws, gp->xt, gp->DP, npad, gp->plan,
                 gp->bop, fit_kl_in_smem(n) ? 1 : 0, fit_early, gp->kern, gp->status,
                 (const int *)nullptr, gp->Wws);  // W kept in global memory as well
      count_launch(2);
    } else {  // one block per problem-objective on the global workspace
      launch_pdl(fit32_kernel<false>, dim3(BM), dim3(fit_threads<false>()),
                 6 * npad * sizeof(float), s, gp->Kh, gp->Kl, Ys, standardize, n, m, gp->Aws,
                 gp->Wws, gp->xt, gp->DP, npad, gp->plan, gp->bop, 0, 0, gp->kern, gp->status,
                 (const int *)nullptr, (float *)nullptr);
      const long long tot = (long long)gp->plan.nwblk * BOUTE_BLKCOLS * gp->plan.nchunk * 32;
      pack_kernel<<<dim3((unsigned)std::min<long long>((tot + 255) / 256, 4096), BM), 256, 0,
                    s>>>(gp->Wws, gp->plan, gp->bop, gp->xt, gp->DP, gp->status);
      count_launch(3);
    }
  } else {
    // the factorisation across many blocks, panel by panel, then alpha across
    // many blocks and the operand images
    const int cap = std::max(1, 2 * sms / BM);
    auto ctas = [&](long long tiles) {
      return (unsigned)std::max(1LL, std::min<long long>(cap, (tiles + kFitbThreads - 1) / kFitbThreads));
    };
    auto grid = [&](long long items) {  // one block per item up to 4 blocks per SM
      return (unsigned)std::max(1LL, std::min<long long>(std::max(1, 4 * sms / BM), items));
    };
    int nl = 0;
    launch_pdl(fitb_load_kernel, dim3(ctas((long long)npad * npad / 2), BM), dim3(kFitbThreads), 0, s,
               (const float *)gp->Kh, n, npad, gp->Aws, gp->fbad);
    ++nl;
    const int nbw = npad / 32;
    for (int p = 0; p < nbw; ++p) {
      const int T = nbw - 1 - p;
      launch_pdl(fitb_diag_kernel, dim3(BM), dim3(64), 0, s, (const float *)gp->Kh, n, npad,
                 gp->Aws, gp->Wws, p, gp->fbad);
      ++nl;
      // items: the panel's block rows below p, then one per (J, chunk) of T_pJ
      const long long items = (long long)T + fitb_t_items(p);
      if (items > 0) {
        launch_pdl(fitb_panel_kernel, dim3(grid(items), BM), dim3(kFitbThreads), 0, s, npad,
                   gp->Aws, (const float *)gp->Wws, p, (const int *)gp->fbad, gp->tpart);
        ++nl;
      }
      // items: W_pJ for J < p, then the trailing tiles
      const long long uitems = (long long)p + (long long)T * (T + 1) / 2;
      if (uitems > 0) {
        launch_pdl(fitb_update_kernel, dim3(grid(uitems), BM), dim3(kFitbThreads), 0, s, npad,
                   gp->Aws, gp->Wws, p, (const int *)gp->fbad, (const float *)gp->tpart);
        ++nl;
      }
    }
    // alpha: W^T (W y) and two refinement steps, each matvec over many blocks
    const int *fb = gp->fbad;
    launch_pdl(fitr_init_kernel, dim3(BM), dim3(256), 0, s, Ys, standardize, n, m, npad,
               gp->fvec, gp->xt, gp->DP, gp->plan, gp->kern, gp->status, fb);
    for (int step = 0; step < 3; ++step) {
      if (step > 0)
        launch_pdl(fitr_resid_kernel, dim3((npad + 15) / 16, BM), dim3(256), 0, s,
                   (const float *)gp->Kh, (const float *)gp->Kl, n, npad, gp->fvec, fb);
      launch_pdl(fitr_wx_kernel, dim3((npad + 7) / 8, BM), dim3(256), 0, s, npad,
                 (const float *)gp->Wws, gp->fvec, step == 0 ? (int)kVy : (int)kVr, fb);
      launch_pdl(fitr_wtx_kernel, dim3(npad / 32, BM), dim3(256), 0, s, npad, n,
                 (const float *)gp->Wws, gp->fvec, step, gp->xt, gp->DP, gp->plan, fb);
      nl += step > 0 ? 3 : 2;
    }
    count_launch(nl + 1);
    const long long tot = (long long)gp->plan.nwblk * BOUTE_BLKCOLS * gp->plan.nchunk * 32;
    pack_kernel<<<dim3((unsigned)std::min<long long>((tot + 255) / 256, 4096), BM), 256, 0, s>>>(
        gp->Wws, gp->plan, gp->bop, gp->xt, gp->DP, gp->status);
    count_launch(1);
  }
  return last_launch_status();
}

int launch_fit(Gp *gp, const double *X, const double *Ys, const double *ls, const double *s2,
               const double *noise, cudaStream_t s) {
  return launch_fit_impl(gp, X, Ys, 0, ls, s2, noise, s);
}

int launch_fit_raw(Gp *gp, const double *X, const double *Y, const double *ls, const double *s2,
                   const double *noise, cudaStream_t s, cudaEvent_t setup_done) {
  return launch_fit_impl(gp, X, Y, 1, ls, s2, noise, s, setup_done);
}

BOUTE_BOUNDS_READER(fit)

}  // namespace boute
