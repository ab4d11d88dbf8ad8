// Noisy acquisition (Sec. 5.2, constrained qNEHVI with q = 1): the
// expectation runs over joint posterior draws of the objectives at the n
// observed points and at the candidate, so the front a candidate improves on
// is itself drawn, sample by sample.
//
// With K = K_nn + sigma^2 I = L L^T, W = L^-1 and the in-sample posterior
// covariance Sigma = K_nn - K_nn K^-1 K_nn = sigma^2 (I - sigma^2 K^-1), a
// joint draw s is the Cholesky factor of the joint covariance (jitter on the
// in-sample block) applied to the normals (z_s, eps_s):
//   f_s(X) = mu_n + F z_s,  F = chol(Sigma + jitter s2 I),  mu_n = y - sigma^2 alpha
//   f_s(x) = mean(x) + l^T z_s + sqrt(cvar) eps_s,  l = F^-1 Sigma_nx
// with Sigma_nx = sigma^2 K^-1 k*. Both per-candidate terms are contractions
// of k*: l^T z_s = k*^T G_s with G = H Z, H = sigma^2 K^-1 F^-T, and
// cvar = k(x,x) - |W k*|^2 - |H^T k*|^2. H^T and G^T therefore become dense
// output blocks of the posterior's tensor-core contraction beside W.
//
//   insample_kernel        one CTA per problem-objective after the fit: K^-1,
//                          F, the in-sample draws, H, G and their operand
//                          images (fp32 arithmetic in shared memory, n <= 128)
//   insample_front_kernel  one warp per (problem, draw): the Pareto front of
//                          the feasible in-sample draws as vertical strips
//   nehvi2_kernel          one thread per candidate: the draws' hypervolume
//                          improvements over their own fronts, averaged
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace boute {

namespace {

constexpr int kInsThreads = 512;

// Row stride of the shared-memory matrices: odd, so that a warp reading one
// column (32 consecutive rows) touches 32 different banks.
__host__ __device__ __forceinline__ int ins_ld(int n) { return n | 1; }
__host__ __device__ __forceinline__ int ins_lda(int n) { return round_up(n, 32) + 4; }
__host__ __device__ __forceinline__ int ins_ldk(int n) { return round_up(n, 32) + 8; }

__device__ __forceinline__ void atomic_max_pos(unsigned *a, float v) {
  atomicMax(a, __float_as_uint(v));  // non-negative floats order as their bits
}

__device__ __forceinline__ int scale_exp(float mx) { return mx > 0.f ? 13 - ilogbf(mx) : 0; }

// Workspace of one problem-objective: F (n x n, zero above the diagonal),
// H^T (n x n), mu_n (n), and max |G| (one word, as float bits).
__host__ __device__ __forceinline__ size_t ins_ws_floats(int n) {
  return 2 * (size_t)n * n + (size_t)n + 4;
}

// The operand image of one output row of a dense block: K positions k, k + 1
// of row `row` of block q, scaled, as fp16 hi/lo pairs (zero beyond n).
__device__ __forceinline__ void pack_dense_pair(const float *src, int n, int k, float scl, int q,
                                                int row, const PostPlan &plan, uint16_t *img) {
  const float v0 = k < n ? src[k] * scl : 0.f, v1 = k + 1 < n ? src[k + 1] * scl : 0.f;
  uint32_t hi, lo;
  split_f16x2(v0, v1, hi, lo);
  const int ncol = plan.ncol[q], cidx = k / BOUTE_ACHUNK;
  uint32_t *blk = (uint32_t *)(img + plan.off[q] + (long long)cidx * 2 * ncol * BOUTE_ACHUNK);
  const int o = sw128_off16(row % BOUTE_BLKCOLS, k % BOUTE_ACHUNK) >> 1;
  const long long base = plan.off[q] + (long long)cidx * 2 * ncol * BOUTE_ACHUNK;
  (void)base;  // (used by the debug build's checks)
  if (BOUTE_INB(base + 2 * ((ncol * BOUTE_ACHUNK >> 1) + o) + 1, plan.image_halves) &&
      BOUTE_INB(k, plan.nchunk * BOUTE_ACHUNK)) {
    blk[o] = hi;
    blk[(ncol * BOUTE_ACHUNK >> 1) + o] = lo;
  }
}

// (1) one CTA per problem-objective: the sequential part. K^-1 = W^T W, the
// jittered in-sample covariance and its Cholesky factor F, H^T = sigma^2
// F^-1 K^-1 by forward substitution; F, H^T and mu_n go to the workspace,
// H^T's operand images and scale exponent to the handle.
__global__ void __launch_bounds__(kInsThreads, 1)
    insample_factor_kernel(const float *Wws, int npad, float *xt, int DP, int nxt,
                           const double *Ys, const double *s2, const double *noise, int n, int m,
                           float *ws, uint16_t *bop, PostPlan plan, int *status) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int bad;
  __shared__ unsigned mxh;
  const int bt = blockIdx.x;
  const int tid = threadIdx.x;
  // row strides: A (L, read along rows by four lanes per row) = 4 mod 32,
  // Kb (K^-1 then H^T, read down columns by eight columns x four k phases)
  // = 8 mod 32, so that neither pattern repeats a bank within a warp
  const int ld = ins_lda(n), ldk = ins_ldk(n);
  float *A = sm, *Kb = A + (size_t)n * ld, *part = Kb + (size_t)n * ldk, *mu = part + 4 * 128;
  const double s2d = s2[bt];
  const double nzd = noise[bt] > 1e-12 * s2d ? noise[bt] : 1e-12 * s2d;  // the fit's floor
  const float sig2 = (float)nzd, jit = (float)(kInsJitter * s2d);
  const int cf = xt_chunk_floats(DP);
  float *x0 = xt + (size_t)bt * nxt * cf;
  float *wsb = ws + (size_t)bt * ins_ws_floats(n);
  pdl_wait();  // the fit's W and alpha
  if (tid == 0) {
    bad = *status == BOUTE_ERR_NOT_PD;
    mxh = 0u;
    wsb[2 * (size_t)n * n + n] = 0.f;  // max |G|, raised by the draws kernel
  }
  // W (lower triangle) and mu_n = y - sigma^2 alpha (alpha = hi + lo)
  const float *W = Wws + (size_t)bt * npad * (npad + 1);
  const int warp = tid >> 5, lane = tid & 31;
  for (int i = warp; i < n; i += kInsThreads / 32) {  // a warp per row, four loads in flight
    float v[kInsMaxN / 32];
#pragma unroll
    for (int r = 0; r < kInsMaxN / 32; ++r) {
      const int k = lane + 32 * r;
      v[r] = k <= i ? W[(size_t)i * (npad + 1) + k] : 0.f;
    }
#pragma unroll
    for (int r = 0; r < kInsMaxN / 32; ++r)
      if (lane + 32 * r < n) A[(size_t)i * ld + lane + 32 * r] = v[r];
  }
  const int b = bt / m, t = bt % m;
  for (int i = tid; i < n; i += kInsThreads) {
    const float *ca = x0 + (size_t)(i / BOUTE_KCHUNK) * cf + xt_alpha_offset(DP) + i % BOUTE_KCHUNK;
    const double al = (double)ca[0] + (double)ca[BOUTE_KCHUNK];
    mu[i] = (float)(Ys[((size_t)b * n + i) * m + t] - nzd * al);
    wsb[2 * (size_t)n * n + i] = mu[i];
  }
  __syncthreads();
  if (bad) return;
  // K^-1 = W^T W: (i, j), j <= i, sum over k >= i of W_ki W_kj (two chains)
  const int npairs = n * (n + 1) / 2;
  for (int e = tid; e < npairs; e += kInsThreads) {
    int i = (int)((sqrtf(8.f * e + 1.f) - 1.f) * 0.5f);
    while (i * (i + 1) / 2 > e) --i;
    while ((i + 1) * (i + 2) / 2 <= e) ++i;
    const int j = e - i * (i + 1) / 2;
    float a0 = 0.f, a1 = 0.f;
    int k = i;
    for (; k + 1 < n; k += 2) {
      a0 = fmaf(A[(size_t)k * ld + i], A[(size_t)k * ld + j], a0);
      a1 = fmaf(A[(size_t)(k + 1) * ld + i], A[(size_t)(k + 1) * ld + j], a1);
    }
    if (k < n) a0 = fmaf(A[(size_t)k * ld + i], A[(size_t)k * ld + j], a0);
    const float acc = a0 + a1;
    Kb[(size_t)i * ldk + j] = acc;
    Kb[(size_t)j * ldk + i] = acc;
  }
  __syncthreads();
  // Sigma + jitter s2 I = sigma^2 (I - sigma^2 K^-1) + jitter s2 I (lower)
  for (int e = tid; e < n * n; e += kInsThreads) {
    const int i = e / n, j = e % n;
    if (j <= i) {
      const float v = sig2 * ((i == j ? 1.f : 0.f) - sig2 * Kb[(size_t)i * ldk + j]);
      A[(size_t)i * ld + j] = i == j ? v + jit : v;
    }
  }
  __syncthreads();
  // Cholesky in 32-column panels: (a) the panel's columns c, rows i >= p0,
  // take the earlier panels' products, A_ic -= sum_{k<p0} L_ik L_ck (a thread
  // holds one row and eight columns c = cg + 4u); (b) warp 0 factors the
  // 32 x 32 diagonal block in registers (lane = row; rows past n are the
  // identity); (c) the rows below solve L_i,panel = A_i,panel L_dd^-T, a
  // thread per row in registers.
  const unsigned FULL = 0xffffffffu;
  const int nb = (n + 31) / 32;
  __shared__ int badp;
  if (tid == 0) badp = 0;
  for (int p = 0; p < nb; ++p) {
    const int p0 = 32 * p, R = n - p0;
    if (p0 > 0) {
      const int ii = tid >> 2, cg = tid & 3;
      if (ii < R) {
        const float *Li = A + (size_t)(p0 + ii) * ld;
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int k = 0; k < p0; ++k) {
          const float l = Li[k];
#pragma unroll
          for (int u = 0; u < 8; ++u) acc[u] = fmaf(l, A[(size_t)(p0 + cg + 4 * u) * ld + k], acc[u]);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (cg + 4 * u <= ii) A[(size_t)(p0 + ii) * ld + p0 + cg + 4 * u] -= acc[u];
      }
      __syncthreads();
    }
    if (warp == 0) {
      // a[k] holds column p0 + c + k of this lane's row: a window that moves
      // one column right every step, so that the step loop keeps static
      // register indices
      const int row = p0 + lane;
      const bool live = row < n;
      float a[32];
#pragma unroll
      for (int k = 0; k < 32; ++k)
        a[k] = (live && k <= lane) ? A[(size_t)row * ld + p0 + k] : (k == lane ? 1.f : 0.f);
      bool okp = true;
      for (int c = 0; c < 32; ++c) {
        const float piv = __shfl_sync(FULL, a[0], c);
        okp = okp && piv > 0.f;
        const float d = sqrtf(fmaxf(piv, 1e-30f));
        const float l = lane == c ? d : (lane > c ? a[0] / d : 0.f);  // L_{lane,c}
#pragma unroll
        for (int k = 1; k < 32; ++k) {
          const float lk = __shfl_sync(FULL, l, (c + k) & 31);  // L_{c+k,c}
          if (c + k < 32 && lane >= c + k) a[k] = fmaf(-l, lk, a[k]);
        }
        if (live && lane >= c) A[(size_t)row * ld + p0 + c] = l;
#pragma unroll
        for (int k = 0; k < 31; ++k) a[k] = a[k + 1];
        a[31] = 0.f;
      }
      if (lane == 0 && !okp) badp = 1;
    }
    __syncthreads();
    if (badp) {  // (uniform)
      if (tid == 0) set_status(status, BOUTE_ERR_NOT_PD);
      return;
    }
    if (tid < R - 32) {
      const int i = p0 + 32 + tid;
      const float *Ld = A + (size_t)p0 * ld + p0;  // L_dd, read as broadcasts
      float bv[32];
#pragma unroll
      for (int c = 0; c < 32; ++c) bv[c] = A[(size_t)i * ld + p0 + c];
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        float sv = bv[c];
#pragma unroll
        for (int k = 0; k < c; ++k) sv = fmaf(-bv[k], Ld[(size_t)c * ld + k], sv);
        bv[c] = sv / Ld[(size_t)c * ld + c];
      }
#pragma unroll
      for (int c = 0; c < 32; ++c) A[(size_t)i * ld + p0 + c] = bv[c];
    }
    __syncthreads();
  }
  for (int e = tid; e < n * n; e += kInsThreads) {  // F, zero above the diagonal
    const int i = e / n, k = e % n;
    wsb[e] = k <= i ? A[(size_t)i * ld + k] : 0.f;
  }
  // H^T = sigma^2 F^-1 K^-1 by forward substitution (in place of K^-1) in
  // blocks of 32 rows: (a) the block's right-hand sides sigma^2 K^-1_rc -
  // sum_{k<r0} F_rk H^T_kc (a thread holds one column and eight rows), then
  // (b) a thread per column solves the block's triangle in registers.
  float hmax = 0.f;
  for (int q = 0; q < nb; ++q) {
    const int r0 = 32 * q;
    {
      const int c = tid & 127, rg = tid >> 7;
      if (c < n) {
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int k = 0; k < r0; ++k) {
          const float hk = Kb[(size_t)k * ldk + c];
#pragma unroll
          for (int u = 0; u < 8; ++u) acc[u] = fmaf(A[(size_t)(r0 + 8 * rg + u) * ld + k], hk, acc[u]);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int r = r0 + 8 * rg + u;
          if (r < n) Kb[(size_t)r * ldk + c] = fmaf(sig2, Kb[(size_t)r * ldk + c], -acc[u]);
        }
      }
    }
    __syncthreads();
    if (tid < n) {
      const int c = tid;
      float hv[32];
#pragma unroll
      for (int rr = 0; rr < 32; ++rr) hv[rr] = r0 + rr < n ? Kb[(size_t)(r0 + rr) * ldk + c] : 0.f;
#pragma unroll
      for (int rr = 0; rr < 32; ++rr) {
        if (r0 + rr < n) {
          const float *Fr = A + (size_t)(r0 + rr) * ld + r0;
          float sv = hv[rr];
#pragma unroll
          for (int k = 0; k < rr; ++k) sv = fmaf(-Fr[k], hv[k], sv);
          hv[rr] = sv / Fr[rr];
          hmax = fmaxf(hmax, fabsf(hv[rr]));
        }
      }
#pragma unroll
      for (int rr = 0; rr < 32; ++rr)
        if (r0 + rr < n) Kb[(size_t)(r0 + rr) * ldk + c] = hv[rr];
    }
    __syncthreads();
  }
  if (tid < n) atomic_max_pos(&mxh, hmax);
  __syncthreads();
  for (int e = tid; e < n * n; e += kInsThreads)
    wsb[(size_t)n * n + e] = Kb[(size_t)(e / n) * ldk + e % n];
  // H^T's operand images (output rows of the H blocks) and scale
  const int eh = scale_exp(__uint_as_float(mxh));
  if (tid == 0) x0[xt_param_offset(DP) + 2 * DP + kParEH] = (float)eh;
  const float sh = exp2i(eh);
  const int kpairs = plan.nchunk * (BOUTE_ACHUNK / 2);
  uint16_t *img = bop + (size_t)bt * plan.image_halves;
  for (int e = tid; e < n * kpairs; e += kInsThreads) {
    const int row = e / kpairs, k = 2 * (e % kpairs);
    pack_dense_pair(Kb + (size_t)row * ldk, n, k, sh, plan.nwblk + row / BOUTE_BLKCOLS, row, plan,
                    img);
  }
}

// (2) the draws, kInsDraws per CTA (grid: draw groups x problem-objectives),
// a warp per draw: Yin[s] = mu_n + F z_s and G^T row s = H^T^T z_s, four
// rows per lane as independent chains; max |G| by atomics.
constexpr int kInsDraws = 4, kDrawThreads = 32 * kInsDraws;

__global__ void __launch_bounds__(kDrawThreads)
    insample_draws_kernel(int n, int S, const float *z, float *Yin, float *gws, float *ws,
                          const int *status) {
  extern __shared__ __align__(16) float sm[];
  const int bt = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ld = ins_ld(n);
  float *F = sm, *Ht = F + (size_t)n * ld, *zs = Ht + (size_t)n * ld, *mu = zs + kInsDraws * kInsMaxN;
  float *wsb = ws + (size_t)bt * ins_ws_floats(n);
  pdl_wait();
  if (*status == BOUTE_ERR_NOT_PD) return;
  for (int i = warp; i < n; i += kInsDraws) {  // a warp per row, eight loads in flight
    float f[kInsMaxN / 32], h[kInsMaxN / 32];
#pragma unroll
    for (int r = 0; r < kInsMaxN / 32; ++r) {
      const int k = lane + 32 * r;
      f[r] = k < n ? wsb[(size_t)i * n + k] : 0.f;
      h[r] = k < n ? wsb[(size_t)n * n + (size_t)i * n + k] : 0.f;
    }
#pragma unroll
    for (int r = 0; r < kInsMaxN / 32; ++r)
      if (lane + 32 * r < n) {
        F[(size_t)i * ld + lane + 32 * r] = f[r];
        Ht[(size_t)i * ld + lane + 32 * r] = h[r];
      }
  }
  for (int i = threadIdx.x; i < n; i += kDrawThreads) mu[i] = wsb[2 * (size_t)n * n + i];
  const int s = blockIdx.x * kInsDraws + warp;
  const size_t zoff = (size_t)bt * S * n;
  float *zw = zs + warp * kInsMaxN;
  if (s < S)
    for (int j = lane; j < n; j += 32) zw[j] = z[zoff + (size_t)s * n + j];
  __syncthreads();
  if (s >= S) return;
  constexpr int R = kInsMaxN / 32;
  float y[R], g[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    y[r] = lane + 32 * r < n ? mu[lane + 32 * r] : 0.f;
    g[r] = 0.f;
  }
  for (int j = 0; j < n; ++j) {
    const float zj = zw[j];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i = lane + 32 * r;
      if (i < n) {
        y[r] = fmaf(F[(size_t)i * ld + j], zj, y[r]);  // zero above the diagonal
        g[r] = fmaf(Ht[(size_t)j * ld + i], zj, g[r]);
      }
    }
  }
  float gm = 0.f;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int i = lane + 32 * r;
    if (i < n && BOUTE_INB(zoff + (long long)s * n + i, (long long)gridDim.y * S * n)) {
      Yin[zoff + (size_t)s * n + i] = y[r];
      gws[zoff + (size_t)s * n + i] = g[r];
      gm = fmaxf(gm, fabsf(g[r]));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) gm = fmaxf(gm, __shfl_xor_sync(0xffffffffu, gm, o));
  if (lane == 0) atomic_max_pos((unsigned *)(wsb + 2 * (size_t)n * n + n), gm);
}

// (3) G^T's operand images (the G blocks) with the scale of max |G|.
__global__ void __launch_bounds__(256)
    insample_pack_kernel(int n, int S, const float *gws, const float *ws, float *xt, int DP,
                         int nxt, uint16_t *bop, PostPlan plan, const int *status) {
  const int bt = blockIdx.y;
  pdl_wait();
  if (*status == BOUTE_ERR_NOT_PD) return;
  const float *wsb = ws + (size_t)bt * ins_ws_floats(n);
  const int eg = scale_exp(wsb[2 * (size_t)n * n + n]);
  if (blockIdx.x == 0 && threadIdx.x == 0)
    xt[(size_t)bt * nxt * xt_chunk_floats(DP) + xt_param_offset(DP) + 2 * DP + kParEG] = (float)eg;
  const float sg = exp2i(eg);
  const int kpairs = plan.nchunk * (BOUTE_ACHUNK / 2);
  uint16_t *img = bop + (size_t)bt * plan.image_halves;
  const float *gb = gws + (size_t)bt * S * n;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < S * kpairs; e += gridDim.x * blockDim.x) {
    const int row = e / kpairs, k = 2 * (e % kpairs);
    pack_dense_pair(gb + (size_t)row * n, n, k, sg, plan.nwblk + plan.nhblk + row / BOUTE_BLKCOLS,
                    row, plan, img);
  }
}

}  // namespace

size_t insample_smem_bytes(int n) {
  return ((size_t)n * (ins_lda(n) + ins_ldk(n)) + 4 * 128 + 128) * sizeof(float);
}

size_t insample_ws_floats(int n) { return ins_ws_floats(n); }

int launch_insample(Gp *gp, const double *Ys, const double *s2, const double *noise,
                    const float *z, float *Yin, cudaStream_t s) {
  const int n = gp->n, BM = gp->B * gp->m, S = gp->plan.S_in;
  if (S < 1 || n > kInsMaxN) return BOUTE_ERR_UNSUPPORTED;
  const size_t smem = insample_smem_bytes(n);
  prefer_shared(insample_factor_kernel);
  cudaFuncSetAttribute(insample_factor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)smem);
  launch_pdl(insample_factor_kernel, dim3(BM), dim3(kInsThreads), smem, s,
             (const float *)gp->Wws, gp->plan.npad, gp->xt, gp->DP, gp->plan.nxt, Ys, s2, noise,
             n, gp->m, gp->iws, gp->bop, gp->plan, gp->status);
  const size_t smem2 = (2 * (size_t)n * ins_ld(n) + kInsDraws * kInsMaxN + kInsMaxN) * sizeof(float);
  prefer_shared(insample_draws_kernel);
  cudaFuncSetAttribute(insample_draws_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)smem2);
  launch_pdl(insample_draws_kernel, dim3((S + kInsDraws - 1) / kInsDraws, BM), dim3(kDrawThreads),
             smem2, s, n, S, z, Yin, gp->gws, gp->iws, (const int *)gp->status);
  const int kpairs = gp->plan.nchunk * (BOUTE_ACHUNK / 2);
  const unsigned gx = (unsigned)std::min(64, (S * kpairs + 255) / 256);
  launch_pdl(insample_pack_kernel, dim3(gx, BM), dim3(256), 0, s, n, S,
             (const float *)gp->gws, (const float *)gp->iws, gp->xt, gp->DP, gp->plan.nxt,
             gp->bop, gp->plan, (const int *)gp->status);
  count_launch(3);
  return last_launch_status();
}

namespace {

constexpr int kFrontPts = kInsMaxN / 32;  // in-sample points per lane
constexpr int kFrontWarps = 4;

// The Pareto front (minimisation) of one draw's feasible in-sample points
// that lie strictly inside the reference box, as the vertical strips of the
// region the front leaves undominated: with the front sorted by f1 (f2 then
// decreasing) q_0 .. q_{P-1},
//   strip 0: (-inf, q_0.f1) x (-inf, r2),  strip i: [q_{i-1}.f1, q_i.f1) x (-inf, q_{i-1}.f2),
//   strip P: [q_{P-1}.f1, r1) x (-inf, q_{P-1}.f2),
// stored as (l1, u1, u2); a point's hypervolume improvement is the sum over
// the strips of (u1 - max(l1, y1))+ (u2 - y2)+. Duplicates keep their lowest
// index, as the front of the observed outcomes does.
__global__ void __launch_bounds__(32 * kFrontWarps)
    insample_front_kernel(const float *Yin, int B, int n, int S, const double *ref,
                          const double *cons, float4 *strips, int *counts) {
  __shared__ float f1s[kFrontWarps][kInsMaxN];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int bs = blockIdx.x * kFrontWarps + w;  // (problem, draw)
  pdl_wait();
  if (bs >= B * S) return;
  const int b = bs / S, s = bs % S;
  const float r1 = (float)ref[(size_t)b * 2], r2 = (float)ref[(size_t)b * 2 + 1];
  const bool hc = cons != nullptr;
  const float c1 = hc ? (float)cons[(size_t)b * 2] : 0.f, c2 = hc ? (float)cons[(size_t)b * 2 + 1] : 0.f;
  const float *y1 = Yin + ((size_t)(b * 2) * S + s) * n, *y2 = Yin + ((size_t)(b * 2 + 1) * S + s) * n;
  float p1[kFrontPts], p2[kFrontPts];
  bool ok[kFrontPts];
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r) {
    const int i = lane + 32 * r;
    ok[r] = i < n;
    p1[r] = ok[r] ? y1[i] : 0.f;
    p2[r] = ok[r] ? y2[i] : 0.f;
    ok[r] = ok[r] && p1[r] < r1 && p2[r] < r2 && (!hc || (p1[r] <= c1 && p2[r] <= c2));
  }
  // dominance: every candidate point against every other (shuffles)
  bool keep[kFrontPts];
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r) keep[r] = ok[r];
#pragma unroll
  for (int r2 = 0; r2 < kFrontPts; ++r2) {
    if (32 * r2 >= n) break;
    for (int src = 0; src < 32; ++src) {
      const float q1 = __shfl_sync(0xffffffffu, p1[r2], src);
      const float q2 = __shfl_sync(0xffffffffu, p2[r2], src);
      const bool qv = __shfl_sync(0xffffffffu, ok[r2] ? 1 : 0, src) != 0;
      const int j = src + 32 * r2;
      if (!qv) continue;
#pragma unroll
      for (int r = 0; r < kFrontPts; ++r) {
        const int i = lane + 32 * r;
        const bool le = q1 <= p1[r] && q2 <= p2[r];
        const bool lt = q1 < p1[r] || q2 < p2[r];
        if (j != i && le && (lt || j < i)) keep[r] = false;  // dominated, or a later duplicate
      }
    }
  }
  // count and rank: on the front f1 values are distinct
  int P = 0;
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r) P += __popc(__ballot_sync(0xffffffffu, keep[r]));
  // compact the front's f1 values into shared memory, then rank by f1
  int base = 0;
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r) {
    const unsigned bal = __ballot_sync(0xffffffffu, keep[r]);
    if (keep[r]) f1s[w][base + __popc(bal & ((1u << lane) - 1u))] = p1[r];
    base += __popc(bal);
  }
  __syncwarp();
  float4 *st = strips + (size_t)bs * (n + 1);
  int rank[kFrontPts];
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r) {
    rank[r] = 0;
    if (keep[r])
      for (int q = 0; q < P; ++q) rank[r] += f1s[w][q] < p1[r] ? 1 : 0;
  }
  __syncwarp();
  // the f1 values in sorted order
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r)
    if (keep[r]) f1s[w][rank[r]] = p1[r];
  __syncwarp();
#pragma unroll
  for (int r = 0; r < kFrontPts; ++r)
    if (keep[r] && BOUTE_INB(rank[r] + 1, n + 1)) {
      const float u1 = rank[r] + 1 < P ? f1s[w][rank[r] + 1] : r1;
      st[rank[r] + 1] = make_float4(p1[r], u1, p2[r], 0.f);
    }
  if (lane == 0) {
    st[0] = make_float4(-INFINITY, P > 0 ? f1s[w][0] : r1, r2, 0.f);
    counts[bs] = P + 1;
  }
}

// One thread per candidate: draw s is y_t = mean_t + shift_t,s + sqrt(cvar_t)
// eps_t,s; with constraints only a feasible draw counts; its improvement is
// summed over draw s's strips. Every thread of a block walks the draws in the
// same order, so a block stages all draws' strips in shared memory once
// (packed, by an exclusive scan of the counts) and reads them as broadcasts;
// when they do not fit it reads them from global memory the same way. VEC:
// the normals load four draws at a time.
constexpr int kAcqThreads = 128;
constexpr int kStripSmem = 3072;  // float4 strips staged per block (48 KB)

template <bool VEC>
__global__ void __launch_bounds__(kAcqThreads)
    nehvi2_kernel(const float *mean, const float *cvar, const float *shift, long long N, int S,
                  const float *eps, long long eps_stride, const float4 *strips, const int *counts,
                  int n, const double *cons, float *acq) {
  extern __shared__ __align__(16) float4 st_s[];
  __shared__ int off_s[kInsMaxS + 1];
  __shared__ int total_s;
  const int b = blockIdx.y;
  const long long c = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  pdl_wait();
  const float4 *stb = strips + (size_t)b * S * (n + 1);
  const int *cnt = counts + (size_t)b * S;
  // exclusive scan of the counts (S <= 1024): loaded by all, scanned by warp 0
  for (int s = threadIdx.x; s < S; s += kAcqThreads) off_s[s + 1] = cnt[s];
  __syncthreads();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int carry = 0;
    for (int base = 0; base < S; base += 32) {
      int v = base + lane < S ? off_s[base + lane + 1] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
      }
      if (base + lane < S) off_s[base + lane + 1] = carry + v;
      carry += __shfl_sync(0xffffffffu, v, 31);
    }
    if (lane == 0) {
      off_s[0] = 0;
      total_s = carry;
    }
  }
  __syncthreads();
  const bool staged = total_s <= kStripSmem;
  if (staged)  // strip q belongs to the draw s with off[s] <= q < off[s + 1]
    for (int q = threadIdx.x; q < total_s; q += kAcqThreads) {
      int lo = 0, hi = S;  // off[lo] <= q < off[hi]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (off_s[mid] <= q) lo = mid;
        else hi = mid;
      }
      if (BOUTE_INB(q - off_s[lo], n + 1)) st_s[q] = stb[(size_t)lo * (n + 1) + (q - off_s[lo])];
    }
  __syncthreads();
  if (c >= N) return;
  const size_t o0 = ((size_t)b * 2) * N + c, o1 = o0 + N;
  const float m0 = mean[o0], m1 = mean[o1];
  const float sd0 = sqrtf(fmaxf(cvar[o0], 0.f)), sd1 = sqrtf(fmaxf(cvar[o1], 0.f));
  const bool hc = cons != nullptr;
  const float c0 = hc ? (float)cons[(size_t)b * 2] : INFINITY;
  const float c1 = hc ? (float)cons[(size_t)b * 2 + 1] : INFINITY;
  const float *e = eps + ((size_t)b * N + c) * eps_stride + (eps_stride == 0 ? (size_t)b * 2 * S : 0);
  const float *sh0 = shift + ((size_t)b * 2) * S * N + c, *sh1 = sh0 + (size_t)S * N;
  // the candidate's normals and its last shift lie inside their arrays
  if (!BOUTE_INB((eps_stride ? ((long long)b * N + c) * eps_stride : (long long)b * 2 * S) + 2 * S - 1,
                 eps_stride ? (long long)gridDim.y * N * eps_stride : (long long)gridDim.y * 2 * S) ||
      !BOUTE_INB((((long long)b * 2 + 1) * S + S - 1) * N + c, (long long)gridDim.y * 2 * S * N))
    return;
  float acc = 0.f;
  auto draw = [&](int s, float e0, float e1, float h0, float h1) {
    const float ya = fmaf(sd0, e0, m0 + h0);
    const float yb = fmaf(sd1, e1, m1 + h1);
    if (!(ya <= c0 && yb <= c1)) return;  // infeasible (or no improvement possible)
    const int k = BOUTE_INB(off_s[s + 1] - off_s[s] - 1, n + 1) ? off_s[s + 1] - off_s[s] : 0;
    const float4 *st = staged ? st_s + off_s[s] : stb + (size_t)s * (n + 1);
    float h = 0.f;
    for (int j = 0; j < k; ++j) {
      const float4 q = st[j];
      const float wdt = fmaxf(q.y - fmaxf(q.x, ya), 0.f), hgt = fmaxf(q.z - yb, 0.f);
      h = fmaf(wdt, hgt, h);
    }
    acc += h;
  };
  // eight draws' shifts and normals are loaded before any is evaluated, so
  // that their latencies overlap
  constexpr int D = 8;
  int s = 0;
  if (VEC) {
    for (; s + D <= S; s += D) {
      float h0[D], h1[D];
#pragma unroll
      for (int u = 0; u < D; ++u) {
        h0[u] = sh0[(size_t)(s + u) * N];
        h1[u] = sh1[(size_t)(s + u) * N];
      }
      float ea[D], eb[D];
#pragma unroll
      for (int u = 0; u < D; u += 4) {
        const float4 a4 = *(const float4 *)(e + s + u), b4 = *(const float4 *)(e + S + s + u);
        ea[u] = a4.x; ea[u + 1] = a4.y; ea[u + 2] = a4.z; ea[u + 3] = a4.w;
        eb[u] = b4.x; eb[u + 1] = b4.y; eb[u + 2] = b4.z; eb[u + 3] = b4.w;
      }
#pragma unroll
      for (int u = 0; u < D; ++u) draw(s + u, ea[u], eb[u], h0[u], h1[u]);
    }
  }
  for (; s < S; ++s) draw(s, e[s], e[S + s], sh0[(size_t)s * N], sh1[(size_t)s * N]);
  if (BOUTE_INB((long long)b * N + c, (long long)gridDim.y * N)) acq[(size_t)b * N + c] = acc / (float)S;
}

}  // namespace

BOUTE_BOUNDS_READER(insample)

int launch_insample_fronts(const float *Yin, int B, int n, int S, const double *ref,
                           const double *cons, float *strips, int *counts, cudaStream_t s) {
  if (n > kInsMaxN) return BOUTE_ERR_UNSUPPORTED;
  const int units = B * S;
  launch_pdl(insample_front_kernel, dim3((units + kFrontWarps - 1) / kFrontWarps),
             dim3(32 * kFrontWarps), 0, s, Yin, B, n, S, ref, cons, (float4 *)strips, counts);
  count_launch();
  return last_launch_status();
}

int launch_nehvi2(const float *mean, const float *cvar, const float *shift, int B, long long N,
                  int S, const float *eps, long long eps_stride, const float *strips,
                  const int *counts, int n, const double *cons, float *acq, cudaStream_t s) {
  const unsigned gx = (unsigned)((N + kAcqThreads - 1) / kAcqThreads);
  const size_t smem = (size_t)kStripSmem * sizeof(float4);
  const bool vec = S % 4 == 0 && eps_stride % 4 == 0 && ((uintptr_t)eps & 15) == 0;
  auto go = [&](auto kern) {
    prefer_shared(kern);
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    launch_pdl(kern, dim3(gx, B), dim3(kAcqThreads), smem, s, mean, cvar, shift, N, S, eps,
               eps_stride, (const float4 *)strips, counts, n, cons, acq);
  };
  if (vec) go(nehvi2_kernel<true>);
  else go(nehvi2_kernel<false>);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
