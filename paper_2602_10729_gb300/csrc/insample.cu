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

constexpr int kInsThreads = 512, kInsWarps = kInsThreads / 32;

// Row stride of the shared-memory matrices: odd, so that a warp reading one
// column (32 consecutive rows) touches 32 different banks.
__host__ __device__ __forceinline__ int ins_ld(int n) { return n | 1; }

__device__ __forceinline__ void atomic_max_pos(unsigned *a, float v) {
  atomicMax(a, __float_as_uint(v));  // non-negative floats order as their bits
}

__device__ __forceinline__ int scale_exp(float mx) { return mx > 0.f ? 13 - ilogbf(mx) : 0; }

__global__ void __launch_bounds__(kInsThreads, 1)
    insample_kernel(const float *Wws, int npad, float *xt, int DP, int nxt, const double *Ys,
                    const double *s2, const double *noise, int n, int m, int S, const float *z,
                    float *Yin, float *gws, uint16_t *bop, PostPlan plan, int *status) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int bad;
  __shared__ unsigned mxh, mxg;
  const int bt = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ld = ins_ld(n);
  float *A = sm, *Kb = A + (size_t)n * ld, *zb = Kb + (size_t)n * ld;
  float *part = zb + (size_t)kInsWarps * n, *mu = part + 4 * 128;
  const double s2d = s2[bt];
  const double nzd = noise[bt] > 1e-12 * s2d ? noise[bt] : 1e-12 * s2d;  // the fit's floor
  const float sig2 = (float)nzd, jit = (float)(kInsJitter * s2d);
  const int cf = xt_chunk_floats(DP);
  float *x0 = xt + (size_t)bt * nxt * cf;
  pdl_wait();  // the fit's W and alpha
  if (tid == 0) {
    bad = *status == BOUTE_ERR_NOT_PD;
    mxh = mxg = 0u;
  }
  // W (lower triangle) and mu_n = y - sigma^2 alpha (alpha = hi + lo)
  const float *W = Wws + (size_t)bt * npad * (npad + 1);
  for (int e = tid; e < n * n; e += kInsThreads) {
    const int i = e / n, k = e % n;
    A[(size_t)i * ld + k] = k <= i ? W[(size_t)i * (npad + 1) + k] : 0.f;
  }
  const int b = bt / m, t = bt % m;
  for (int i = tid; i < n; i += kInsThreads) {
    const float *ca = x0 + (size_t)(i / BOUTE_KCHUNK) * cf + xt_alpha_offset(DP) + i % BOUTE_KCHUNK;
    const double al = (double)ca[0] + (double)ca[BOUTE_KCHUNK];
    mu[i] = (float)(Ys[((size_t)b * n + i) * m + t] - nzd * al);
  }
  __syncthreads();
  if (bad) return;
  // K^-1 = W^T W: (i, j), j <= i, sum over k >= i of W_ki W_kj
  const int npairs = n * (n + 1) / 2;
  for (int e = tid; e < npairs; e += kInsThreads) {
    int i = (int)((sqrtf(8.f * e + 1.f) - 1.f) * 0.5f);
    while (i * (i + 1) / 2 > e) --i;
    while ((i + 1) * (i + 2) / 2 <= e) ++i;
    const int j = e - i * (i + 1) / 2;
    float acc = 0.f;
    for (int k = i; k < n; ++k) acc = fmaf(A[(size_t)k * ld + i], A[(size_t)k * ld + j], acc);
    Kb[(size_t)i * ld + j] = acc;
    Kb[(size_t)j * ld + i] = acc;
  }
  __syncthreads();
  // Sigma + jitter s2 I = sigma^2 (I - sigma^2 K^-1) + jitter s2 I (lower)
  for (int e = tid; e < n * n; e += kInsThreads) {
    const int i = e / n, j = e % n;
    if (j <= i) {
      const float v = sig2 * ((i == j ? 1.f : 0.f) - sig2 * Kb[(size_t)i * ld + j]);
      A[(size_t)i * ld + j] = i == j ? v + jit : v;
    }
  }
  __syncthreads();
  // Cholesky, right-looking on the unscaled columns: step k subtracts
  // a_ik a_jk / a_kk from the trailing block; column k and the pivot are
  // final after step k and are scaled once at the end (one barrier a step)
  for (int k = 0; k < n; ++k) {
    const float dk = A[(size_t)k * ld + k];
    if (!(dk > 0.f)) {  // every thread reads the same pivot
      if (tid == 0) set_status(status, BOUTE_ERR_NOT_PD);
      return;
    }
    const float rdk = 1.f / dk;
    const int r = n - 1 - k;
    for (int e = tid; e < r * r; e += kInsThreads) {
      const int i = k + 1 + e / r, j = k + 1 + e % r;
      if (j <= i)
        A[(size_t)i * ld + j] =
            fmaf(-A[(size_t)i * ld + k] * rdk, A[(size_t)j * ld + k], A[(size_t)i * ld + j]);
    }
    __syncthreads();
  }
  for (int e = tid; e < n * n; e += kInsThreads) {
    const int i = e / n, k = e % n;
    if (k < i) A[(size_t)i * ld + k] = A[(size_t)i * ld + k] / sqrtf(A[(size_t)k * ld + k]);
  }
  __syncthreads();
  for (int k = tid; k < n; k += kInsThreads) A[(size_t)k * ld + k] = sqrtf(A[(size_t)k * ld + k]);
  __syncthreads();
  // the in-sample draws: Yin[s] = mu_n + F z_s (a warp per draw)
  const size_t zoff = (size_t)bt * S * n;
  float *zw = zb + (size_t)warp * n;
  for (int s = warp; s < S; s += kInsWarps) {
    for (int j = lane; j < n; j += 32) zw[j] = z[zoff + (size_t)s * n + j];
    __syncwarp();
    for (int i = lane; i < n; i += 32) {
      float v = mu[i];
      const float *fr = A + (size_t)i * ld;
      for (int j = 0; j <= i; ++j) v = fmaf(fr[j], zw[j], v);
      Yin[zoff + (size_t)s * n + i] = v;
    }
    __syncwarp();
  }
  // H^T = sigma^2 F^-1 K^-1 by forward substitution, in place of K^-1, row by
  // row: thread (part, c) sums every fourth k of F_rk H^T_kc
  const int c = tid & 127, pp = tid >> 7;
  for (int r = 0; r < n; ++r) {
    float acc = 0.f;
    if (c < n)
      for (int k = pp; k < r; k += 4) acc = fmaf(A[(size_t)r * ld + k], Kb[(size_t)k * ld + c], acc);
    part[pp * 128 + c] = acc;
    __syncthreads();
    if (pp == 0 && c < n) {
      const float sum = (part[c] + part[128 + c]) + (part[256 + c] + part[384 + c]);
      const float h = (sig2 * Kb[(size_t)r * ld + c] - sum) / A[(size_t)r * ld + r];
      Kb[(size_t)r * ld + c] = h;
      atomic_max_pos(&mxh, fabsf(h));
    }
    __syncthreads();
  }
  // G^T = (H Z)^T: row s, G_js = sum_c H^T_cj z_s,c (a warp per draw)
  float gmax = 0.f;
  const size_t goff = (size_t)bt * S * n;
  for (int s = warp; s < S; s += kInsWarps) {
    for (int j = lane; j < n; j += 32) zw[j] = z[zoff + (size_t)s * n + j];
    __syncwarp();
    for (int j = lane; j < n; j += 32) {
      float g = 0.f;
      for (int cc = 0; cc < n; ++cc) g = fmaf(Kb[(size_t)cc * ld + j], zw[cc], g);
      gws[goff + (size_t)s * n + j] = g;
      gmax = fmaxf(gmax, fabsf(g));
    }
    __syncwarp();
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, o));
  if (lane == 0) atomic_max_pos(&mxg, gmax);
  __syncthreads();  // (also makes this block's writes of gws visible to it)
  const int eh = scale_exp(__uint_as_float(mxh)), eg = scale_exp(__uint_as_float(mxg));
  if (tid == 0) {  // the epilogue's scales (chunk 0's parameters)
    float *par = x0 + xt_param_offset(DP) + 2 * DP;
    par[kParEH] = (float)eh;
    par[kParEG] = (float)eg;
  }
  // operand images: output row R < n is H^T row R (the H blocks), R >= n is
  // G^T row R - n (the G blocks); pairs of K positions, zero beyond n
  const float sh = exp2i(eh), sg = exp2i(eg);
  const int kpairs = plan.nchunk * (BOUTE_ACHUNK / 2);
  uint16_t *img = bop + (size_t)bt * plan.image_halves;
  const long long tot = (long long)(n + S) * kpairs;
  for (long long e = tid; e < tot; e += kInsThreads) {
    const int R = (int)(e / kpairs), k = 2 * (int)(e % kpairs);
    const bool hrow = R < n;
    const int row = hrow ? R : R - n;
    const float *src = hrow ? Kb + (size_t)row * ld : gws + goff + (size_t)row * n;
    const float scl = hrow ? sh : sg;
    const float v0 = k < n ? src[k] * scl : 0.f, v1 = k + 1 < n ? src[k + 1] * scl : 0.f;
    uint32_t hi, lo;
    split_f16x2(v0, v1, hi, lo);
    const int q = (hrow ? plan.nwblk : plan.nwblk + plan.nhblk) + row / BOUTE_BLKCOLS;
    const int ncol = plan.ncol[q], cidx = k / BOUTE_ACHUNK;
    uint32_t *blk = (uint32_t *)(img + plan.off[q] + (long long)cidx * 2 * ncol * BOUTE_ACHUNK);
    const int o = sw128_off16(row % BOUTE_BLKCOLS, k % BOUTE_ACHUNK) >> 1;
    blk[o] = hi;
    blk[(ncol * BOUTE_ACHUNK >> 1) + o] = lo;
  }
}

}  // namespace

size_t insample_smem_bytes(int n) {
  return (2 * (size_t)n * ins_ld(n) + (size_t)kInsWarps * n + 4 * 128 + 128) * sizeof(float);
}

int launch_insample(Gp *gp, const double *Ys, const double *s2, const double *noise,
                    const float *z, float *Yin, cudaStream_t s) {
  const int n = gp->n, BM = gp->B * gp->m;
  if (gp->plan.S_in < 1 || n > kInsMaxN) return BOUTE_ERR_UNSUPPORTED;
  const size_t smem = insample_smem_bytes(n);
  prefer_shared(insample_kernel);
  cudaFuncSetAttribute(insample_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  launch_pdl(insample_kernel, dim3(BM), dim3(kInsThreads), smem, s, (const float *)gp->Wws,
             gp->plan.npad, gp->xt, gp->DP, gp->plan.nxt, Ys, s2, noise, n, gp->m,
             gp->plan.S_in, z, Yin, gp->gws, gp->bop, gp->plan, gp->status);
  count_launch();
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
    if (keep[r]) {
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
// summed over draw s's strips (read as warp-wide broadcasts).
__global__ void __launch_bounds__(256)
    nehvi2_kernel(const float *mean, const float *cvar, const float *shift, long long N, int S,
                  const float *eps, long long eps_stride, const float4 *strips, const int *counts,
                  int n, const double *cons, float *acq) {
  const int b = blockIdx.y;
  const long long c = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  pdl_wait();
  if (c >= N) return;
  const size_t o0 = ((size_t)b * 2) * N + c, o1 = o0 + N;
  const float m0 = mean[o0], m1 = mean[o1];
  const float sd0 = sqrtf(fmaxf(cvar[o0], 0.f)), sd1 = sqrtf(fmaxf(cvar[o1], 0.f));
  const bool hc = cons != nullptr;
  const float c0 = hc ? (float)cons[(size_t)b * 2] : 0.f, c1 = hc ? (float)cons[(size_t)b * 2 + 1] : 0.f;
  const float *e = eps + ((size_t)b * N + c) * eps_stride + (eps_stride == 0 ? (size_t)b * 2 * S : 0);
  const float *sh0 = shift + ((size_t)b * 2) * S * N + c, *sh1 = sh0 + (size_t)S * N;
  const float4 *stb = strips + (size_t)b * S * (n + 1);
  const int *cnt = counts + (size_t)b * S;
  float acc = 0.f;
  for (int s = 0; s < S; ++s) {
    const float ya = fmaf(sd0, e[s], m0 + sh0[(size_t)s * N]);
    const float yb = fmaf(sd1, e[S + s], m1 + sh1[(size_t)s * N]);
    if (hc && !(ya <= c0 && yb <= c1)) continue;
    const float4 *st = stb + (size_t)s * (n + 1);
    const int k = cnt[s];
    float h = 0.f;
    for (int j = 0; j < k; ++j) {
      const float4 q = st[j];
      const float wdt = q.y - fmaxf(q.x, ya), hgt = q.z - yb;
      if (wdt > 0.f && hgt > 0.f) h = fmaf(wdt, hgt, h);
    }
    acc += h;
  }
  acq[(size_t)b * N + c] = acc / (float)S;
}

}  // namespace

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
  const unsigned gx = (unsigned)((N + 255) / 256);
  launch_pdl(nehvi2_kernel, dim3(gx, B), dim3(256), 0, s, mean, cvar, shift, N, S, eps,
             eps_stride, (const float4 *)strips, counts, n, cons, acq);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
