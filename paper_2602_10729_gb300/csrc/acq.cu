// Acquisition kernels: closed-form 2-objective EHVI and Monte-Carlo
// hypervolume improvement over the box decomposition of the front.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "internal.h"
#include "mc2.cuh"
#include "warp_select.cuh"

namespace boute {

namespace {

constexpr float kInvSqrt2Pi = 0.3989422804014327f;
constexpr float kInvSqrt2 = 0.7071067811865476f;

// Small part of psi: with z = (x - mu)/sigma, E[(x - Y)_+] = max(x - mu, 0) +
// sigma * gm(z), gm(z) = phi(|z|) - |z| Phi(-|z|) >= 0 (the identity
// G(z) = z + G(-z) for G(z) = z Phi(z) + phi(z)). Keeping the linear part
// apart avoids cancellation for points far to either side of x. In the tail
// the difference itself cancels (gm ~ phi(t) / t^2), so for t >= 3 it is
// taken from Laplace's continued fraction of the Mills ratio Phi(-t) / phi(t)
// = 1 / x_0, x_k = t + (k + 1) / x_{k+1}: gm = phi(t) (1 - t / x_0) =
// phi(t) / (x_0 x_1). Truncated at x_12 = t, the fraction is the rational
// function P(t^2) / Q(t^2) below (positive coefficients, no cancellation),
// within 1.2e-6 of gm / phi for t >= 3. The rounding of t^2 in phi's
// exponent is recovered by an fma. |z| is capped where gm is already zero,
// so that infinite z gives 0, not NaN.
__device__ __forceinline__ float gm(float z) {
  const float t = fminf(fabsf(z), 1.0e4f);
  const float h = t * t, l = fmaf(t, t, -h);  // t^2 = h + l exactly
  const float phi = expf(-0.5f * h) * fmaf(-0.5f, l, 1.0f) * kInvSqrt2Pi;
  if (t < 3.0f) return phi - t * (0.5f * erfcf(t * kInvSqrt2));
  if (t >= 14.0f) return 0.f;  // (phi(14) is below the fp32 range)
  float p = h + 75.f;
  p = fmaf(p, h, 1926.f);
  p = fmaf(p, h, 20370.f);
  p = fmaf(p, h, 82845.f);
  p = fmaf(p, h, 89055.f);
  float q = h + 78.f;
  q = fmaf(q, h, 2145.f);
  q = fmaf(q, h, 25740.f);
  q = fmaf(q, h, 135135.f);
  q = fmaf(q, h, 270270.f);
  q = fmaf(q, h, 135135.f);
  return phi * __fdividef(p, q);
}

__device__ __forceinline__ float std_cdf(float z) { return 0.5f * erfcf(-z * kInvSqrt2); }

// A threshold as a finite float (an infinite threshold constrains nothing:
// FLT_MAX is above every finite value and keeps the differences below finite).
__device__ __forceinline__ float threshold(double c) {
  return fminf(fmaxf((float)c, -FLT_MAX), FLT_MAX);
}

// ---- closed-form EHVI, m = 2 ---------------------------------------------------
// Cells i = 0..P of the front sorted by f1: f1 in [a_i, b_i), f2 below u_i,
// a_0 = -inf, b_P = r1, u_0 = r2. EHVI = sum_i [psi1(b_i) - psi1(a_i)] psi2(u_i).
// CONS (Sec. 5.2, constrained qNEHVI, thresholds k_t on the minimised
// objectives, cons: B x 2): psi_t becomes psi_t^c(v) = E[(v - Y)_+ 1[Y <= k_t]],
// which is psi_t(min(v, k_t)) + (v - k_t)_+ Phi((k_t - mu_t) / sigma_t), since
// below k_t the indicator is one and above it (v - Y) splits into (k_t - Y) +
// (v - k_t). Per cell psi1^c(b) - psi1^c(a) is then the unconstrained
// difference between the clamped bounds plus (max(b, k1) - max(a, k1)) Phi_1.
template <bool CONS>
__global__ void __launch_bounds__(256) ehvi2d_kernel(const float *mean, const float *var,
                                                     long long N, const double *front,
                                                     const int *P, int n, const double *ref,
                                                     const double *cons, float *acq) {
  extern __shared__ float cells[];  // bnd[n+1] (b_i), up[n+1] (u_i)
  pdl_wait();
  const int b = blockIdx.y;
  const int Pb = P[b];
  float *bnd = cells, *up = cells + (n + 1);
  const double *F = front + (size_t)b * n * 2;
  const float r1 = (float)ref[2 * b], r2 = (float)ref[2 * b + 1];
  const float k1 = CONS ? threshold(cons[2 * b]) : 0.f, k2 = CONS ? threshold(cons[2 * b + 1]) : 0.f;
  for (int i = threadIdx.x; i <= Pb; i += blockDim.x) {
    bnd[i] = i == Pb ? r1 : (float)F[2 * i];
    up[i] = i == 0 ? r2 : (float)F[2 * (i - 1) + 1];
  }
  __syncthreads();
  const float *m1 = mean + (size_t)b * 2 * N, *m2 = m1 + N;
  const float *v1 = var + (size_t)b * 2 * N, *v2 = v1 + N;
  for (long long c = (long long)blockIdx.x * blockDim.x + threadIdx.x; c < N;
       c += (long long)gridDim.x * blockDim.x) {
    const float mu1 = m1[c], mu2 = m2[c];
    const float sg1 = sqrtf(fmaxf(v1[c], 0.f)), sg2 = sqrtf(fmaxf(v2[c], 0.f));
    const float is1 = sg1 > 0.f ? 1.f / sg1 : 0.f, is2 = sg2 > 0.f ? 1.f / sg2 : 0.f;
    // CONS: P(Y_t <= k_t) (a step when sigma_t = 0) and max(a, k1) of cell 0
    float F1 = 1.f, F2 = 1.f, ahi = k1;
    if (CONS) {
      F1 = sg1 > 0.f ? std_cdf((k1 - mu1) * is1) : (mu1 <= k1 ? 1.f : 0.f);
      F2 = sg2 > 0.f ? std_cdf((k2 - mu2) * is2) : (mu2 <= k2 ? 1.f : 0.f);
    }
    float e = 0.f, ga = 0.f, a = -INFINITY;
    for (int i = 0; i <= Pb; ++i) {
      const float bb = CONS ? fminf(bnd[i], k1) : bnd[i], u = CONS ? fminf(up[i], k2) : up[i];
      const float gb = sg1 > 0.f ? gm((bb - mu1) * is1) : 0.f;
      const float lin = mu1 <= a ? bb - a : (mu1 <= bb ? bb - mu1 : 0.f);
      float D = fmaxf(fmaf(sg1, gb - ga, lin), 0.f);
      const float g2 = sg2 > 0.f ? gm((u - mu2) * is2) : 0.f;
      float psi2 = fmaf(sg2, g2, fmaxf(u - mu2, 0.f));
      if (CONS) {
        const float bhi = fmaxf(bnd[i], k1);
        D = fmaf(bhi - ahi, F1, D);
        ahi = bhi;
        psi2 = fmaf(fmaxf(up[i] - k2, 0.f), F2, psi2);
      }
      e = fmaf(D, psi2, e);
      ga = gb;
      a = bb;
    }
    if (BOUTE_INB((long long)b * N + c, (long long)gridDim.y * N)) acq[(size_t)b * N + c] = e;
  }
}

// ---- Monte-Carlo HVI: one warp per candidate, lanes over samples ---------------
// Each sample's HVI is the volume of [y, ref] inside the disjoint boxes:
// sum_k prod_t (u_kt - max(l_kt, y_t))_+.
// CONS: a sample with some y_t above its threshold (cons: B x M) counts zero
// (its first coordinate is moved beyond every box).
//
// With S a multiple of 128 up to 256 every lane holds its 4 S / 128 samples
// of the candidate in registers, and each box is visited once per candidate:
// its lower bounds are raised to the candidate's smallest sample per
// objective (no sample lies below them), which makes every box finite,
// w_t = u_t - l'_t, and a box with some w_t <= 0 (every sample at or above
// its upper bound) is skipped by the whole warp; otherwise each sample adds
// prod_t w_t * prod_t sat((u_t - y_t) / w_t), since (u - max(l', y))_+ =
// w sat((u - y) / w) for y >= l': one saturating fma per objective.
template <int M, bool CONS, int NV>
__device__ __forceinline__ float mc_hvi_regs(const float *e, int S, const float (&mu)[M],
                                             const float (&sg)[M], const float (&kc)[M],
                                             const float *lo, const float *hi, int K, int lane,
                                             float4 *stage) {
  static_assert(M <= 3, "a box's constants fit two float4");
  constexpr int NS = 4 * NV;
  float y[NS][M];
#pragma unroll
  for (int v = 0; v < NV; ++v)
#pragma unroll
    for (int t = 0; t < M; ++t) {
      const float4 z = __ldcs((const float4 *)(e + (size_t)t * S + 128 * v + 4 * lane));
      y[4 * v][t] = fmaf(sg[t], z.x, mu[t]);
      y[4 * v + 1][t] = fmaf(sg[t], z.y, mu[t]);
      y[4 * v + 2][t] = fmaf(sg[t], z.z, mu[t]);
      y[4 * v + 3][t] = fmaf(sg[t], z.w, mu[t]);
    }
  float ymin[M];
#pragma unroll
  for (int t = 0; t < M; ++t) {
    float v = y[0][t];
#pragma unroll
    for (int j = 1; j < NS; ++j) v = fminf(v, y[j][t]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    ymin[t] = v;
  }
  if (CONS) {
#pragma unroll
    for (int j = 0; j < NS; ++j) {
      bool ok = true;
#pragma unroll
      for (int t = 0; t < M; ++t) ok = ok && y[j][t] <= kc[t];
      if (!ok) y[j][0] = kInfeasible;
    }
  }
  // the products and the sum over pairs of samples in packed f32x2 (the
  // saturating fmas have no packed form): two partial sums per lane. The
  // boxes' constants (1/w_t, u_t/w_t, prod w_t) are formed 32 boxes at a time,
  // one box per lane, and staged in this warp's 64 float4 of shared memory;
  // the live boxes are then visited in order, their constants read back by
  // broadcast
  unsigned long long sum2 = 0ull;
  for (int k0 = 0; k0 < K; k0 += 32) {
    const int kb = k0 + lane;
    float cw[3] = {0.f, 0.f, 0.f}, ch[3] = {0.f, 0.f, 0.f}, Wb = 0.f;
    bool lv = false;
    if (kb < K) {
      lv = true;
      Wb = 1.f;
#pragma unroll
      for (int t = 0; t < M; ++t) {
        const float h = hi[kb * M + t];
        const float w = h - fmaxf(lo[kb * M + t], ymin[t]);
        lv = lv && w > 0.f;
        cw[t] = rcp_fast(w);  // (relative error ~2^-23; the clamp absorbs it at the edges)
        ch[t] = h * cw[t];
        Wb *= w;
      }
    }
    __syncwarp();  // the previous group's constants are read
    stage[lane] = make_float4(cw[0], cw[1], cw[2], Wb);
    stage[32 + lane] = make_float4(ch[0], ch[1], ch[2], 0.f);
    __syncwarp();
    unsigned todo = __ballot_sync(0xffffffffu, lv);
    while (todo) {
      const int jb = __ffs(todo) - 1;
      todo &= todo - 1;
      const float4 ca = stage[jb], cb = stage[32 + jb];
      const float iw[3] = {ca.x, ca.y, ca.z}, hw[3] = {cb.x, cb.y, cb.z};
      const unsigned long long W2 = f2_dup(ca.w);
#pragma unroll
      for (int j = 0; j < NS; j += 2) {
        unsigned long long p = f2_pack(fma_sat(-y[j][0], iw[0], hw[0]),
                                       fma_sat(-y[j + 1][0], iw[0], hw[0]));
#pragma unroll
        for (int t = 1; t < M; ++t)
          p = f2_mul(p, f2_pack(fma_sat(-y[j][t], iw[t], hw[t]),
                                fma_sat(-y[j + 1][t], iw[t], hw[t])));
        sum2 = f2_fma(W2, p, sum2);
      }
    }
  }
  float s0, s1;
  f2_split(sum2, s0, s1);
  return s0 + s1;
}

template <int M, bool CONS>
__global__ void __launch_bounds__(512) mchvi_kernel(const float *mean, const float *var, int B,
                                                    long long N, const float *lower,
                                                    const float *upper, const int *Kc,
                                                    int box_cap, const float *eps, int S,
                                                    long long eps_stride, const double *cons,
                                                    float *acq) {
  extern __shared__ float boxes[];  // per problem in this block: lo[K][M], hi[K][M]
  __shared__ float4 stage[16][64];  // per warp: 32 boxes' constants (mc_hvi_regs)
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int b = blockIdx.y;
  const int K = BOUTE_INB(Kc[b], box_cap + 1) ? Kc[b] : 0;
  float *lo = boxes, *hi = boxes + (size_t)box_cap * M;
  for (int i = threadIdx.x; i < K * M; i += blockDim.x) {
    lo[i] = lower[(size_t)b * box_cap * M + i];
    hi[i] = upper[(size_t)b * box_cap * M + i];
  }
  __syncthreads();
  float kc[M];
#pragma unroll
  for (int t = 0; t < M; ++t) kc[t] = CONS ? threshold(cons[(size_t)b * M + t]) : 0.f;
  const float *mb = mean + (size_t)b * M * N, *vb = var + (size_t)b * M * N;
  const bool vec = (S % 128) == 0 && ((uintptr_t)eps & 15) == 0 && (eps_stride % 4) == 0;
  for (long long c = (long long)blockIdx.x * wpb + warp; c < N; c += (long long)gridDim.x * wpb) {
    float mu[M], sg[M];
#pragma unroll
    for (int t = 0; t < M; ++t) {
      mu[t] = mb[(size_t)t * N + c];
      sg[t] = sqrtf(fmaxf(vb[(size_t)t * N + c], 0.f));
    }
    const float *e = eps + ((size_t)b * N + c) * eps_stride +
                     (eps_stride == 0 ? (size_t)b * M * S : 0);
    if (!BOUTE_INB((eps_stride ? ((long long)b * N + c) * eps_stride : (long long)b * M * S) +
                       M * S - 1,
                   eps_stride ? (long long)B * N * eps_stride : (long long)B * M * S))
      continue;  // (warp-uniform)
    float sum = 0.f;
    if (vec && S == 256) {
      sum = mc_hvi_regs<M, CONS, 2>(e, S, mu, sg, kc, lo, hi, K, lane, stage[warp]);
    } else if (vec && S == 128) {
      sum = mc_hvi_regs<M, CONS, 1>(e, S, mu, sg, kc, lo, hi, K, lane, stage[warp]);
    } else if (vec) {
      for (int s0 = 4 * lane; s0 < S; s0 += 128) {
        float4 z[M];
#pragma unroll
        for (int t = 0; t < M; ++t) z[t] = __ldcs((const float4 *)(e + (size_t)t * S + s0));
        float y[4][M];
#pragma unroll
        for (int t = 0; t < M; ++t) {
          y[0][t] = fmaf(sg[t], z[t].x, mu[t]);
          y[1][t] = fmaf(sg[t], z[t].y, mu[t]);
          y[2][t] = fmaf(sg[t], z[t].z, mu[t]);
          y[3][t] = fmaf(sg[t], z[t].w, mu[t]);
        }
        if (CONS) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            bool ok = true;
#pragma unroll
            for (int t = 0; t < M; ++t) ok = ok && y[j][t] <= kc[t];
            if (!ok) y[j][0] = kInfeasible;
          }
        }
        for (int k = 0; k < K; ++k) {
          float l[M], h[M];
#pragma unroll
          for (int t = 0; t < M; ++t) {
            l[t] = lo[k * M + t];
            h[t] = hi[k * M + t];
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            float v = fmaxf(h[0] - fmaxf(l[0], y[j][0]), 0.f);
#pragma unroll
            for (int t = 1; t < M; ++t) v *= fmaxf(h[t] - fmaxf(l[t], y[j][t]), 0.f);
            sum += v;
          }
        }
      }
    } else {
      for (int s = lane; s < S; s += 32) {
        float y[M];
#pragma unroll
        for (int t = 0; t < M; ++t) y[t] = fmaf(sg[t], e[(size_t)t * S + s], mu[t]);
        if (CONS) {
          bool ok = true;
#pragma unroll
          for (int t = 0; t < M; ++t) ok = ok && y[t] <= kc[t];
          if (!ok) y[0] = kInfeasible;
        }
        for (int k = 0; k < K; ++k) {
          float v = fmaxf(hi[k * M] - fmaxf(lo[k * M], y[0]), 0.f);
#pragma unroll
          for (int t = 1; t < M; ++t) v *= fmaxf(hi[k * M + t] - fmaxf(lo[k * M + t], y[t]), 0.f);
          sum += v;
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0 && BOUTE_INB((long long)b * N + c, (long long)B * N))
      acq[(size_t)b * N + c] = sum / (float)S;
  }
}

// 2-objective Monte-Carlo HVI over the strip decomposition (mc2.cuh): one
// warp per candidate, a float4 of base normals per lane and objective when
// S = 128.
// SEL: also select the ksel <= 32 best candidates of each problem as they are
// scored: every warp keeps a running top-32 of its candidates, each block
// merges its warps' lists into sel_keys, and the last block of a problem to
// finish (sel_cnt) merges all the blocks' lists, writes idx / val and sets
// the counter back to zero.
// CONS: samples above a threshold (cons: B x 2) count zero.
constexpr int kSelGroup = 32;  // blocks per selection group

template <bool SEL, bool CONS>
__global__ void __launch_bounds__(512, 2) mchvi2_kernel(const float *mean, const float *var,
                                                     long long N, const float *lower,
                                                     const float *upper, const int *Kc,
                                                     int box_cap, const float *eps, int S,
                                                     long long eps_stride, const double *cons,
                                                     float *acq, int ksel,
                                                     unsigned long long *sel_keys,
                                                     long long *idx, float *val) {
  // k >= 1: (b/D, 1/D, u, D); [0]: (b_0, u_0, -, -); then zero strips up to
  // 1 + a multiple of 4 (they add exactly nothing), box_cap + 4 in all
  extern __shared__ float4 strips4[];
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  const int b = blockIdx.y;
  const int K = mc2_load_strips(strips4, lower, upper, Kc, b, box_cap, threadIdx.x, blockDim.x);
  const int Kp = mc2_padded(K);
  __syncthreads();
  const float k1 = CONS ? threshold(cons[2 * b]) : 0.f, k2 = CONS ? threshold(cons[2 * b + 1]) : 0.f;
  const float *m1 = mean + (size_t)b * 2 * N, *m2 = m1 + N;
  const float *v1 = var + (size_t)b * 2 * N, *v2 = v1 + N;
  const bool vec = (S == 128) && ((uintptr_t)eps & 15) == 0 && (eps_stride % 4) == 0;
  const long long cstride = (long long)gridDim.x * wpb;
  const float inv_s = 1.f / (float)S;
  WarpTopBatch sel;  // this warp's running top-32 (SEL)
  auto eps_of = [&](long long c) {
    return eps + ((size_t)b * N + c) * eps_stride + (eps_stride == 0 ? (size_t)b * 2 * S : 0);
  };
  // improvement of one sample (the direct strip sum)
  auto hvi = [&](float y1, float y2) {
    float acc = 0.f;
    if (K > 0) {
      const float4 t = strips4[0];
      acc = fmaxf(t.x - y1, 0.f) * fmaxf(t.y - y2, 0.f);
    }
    for (int k = 1; k < K; ++k) {
      const float4 t = strips4[k];
      const float w = fma_sat(-y1, t.y, t.x);
      acc = fmaf(w * t.w, fmaxf(t.z - y2, 0.f), acc);
    }
    return acc;
  };
  if (vec) {
    // S = 128: one float4 per lane per objective; the next candidate's
    // samples and posterior are loaded before this one is scored
    // (B N < 2^31: candidate indices in 32 bits; the samples' pointer advances
    // by a fixed step; the last prefetch repeats the current candidate)
    const int Ni = (int)N, cs = (int)cstride;
    int c = blockIdx.x * wpb + warp;
    const size_t estep = (size_t)cs * eps_stride;
    const float *ep = eps_of(c < Ni ? c : 0) + 4 * lane;
    float4 z1 = make_float4(0.f, 0.f, 0.f, 0.f), z2 = z1;
    float pm1 = 0.f, pm2 = 0.f, pv1 = 0.f, pv2 = 0.f;
    if (c < Ni) {
      z1 = __ldcs((const float4 *)ep);
      z2 = __ldcs((const float4 *)(ep + S));
      pm1 = m1[c]; pm2 = m2[c]; pv1 = v1[c]; pv2 = v2[c];
    }
    const float4 t0 = K > 0 ? strips4[0] : make_float4(0.f, 0.f, 0.f, 0.f);
    for (; c < Ni; c += cs) {
      const float4 c1 = z1, c2 = z2;
      const float mu1 = pm1, mu2 = pm2, qv1 = pv1, qv2 = pv2;
      const bool more = c + cs < Ni;
      const int cn = more ? c + cs : c;
      ep = more ? ep + estep : ep;
      z1 = __ldcs((const float4 *)ep);
      z2 = __ldcs((const float4 *)(ep + S));
      pm1 = m1[cn]; pm2 = m2[cn]; pv1 = v1[cn]; pv2 = v2[cn];
      const float sum =
          mc2_warp_total(mc2_lane_sum<CONS>(strips4, K, Kp, t0, c1, c2, mu1, mu2, qv1, qv2, k1, k2));
      if (lane == 0 && BOUTE_INB((long long)b * N + c, (long long)gridDim.y * N))
        acq[(size_t)b * N + c] = sum * inv_s;
      if (SEL) sel.add(make_key(sum * inv_s, (unsigned)c), lane);
    }
  } else {
  for (long long c = (long long)blockIdx.x * wpb + warp; c < N; c += cstride) {
    const float mu1 = m1[c], mu2 = m2[c];
    const float sg1 = sqrt_fast(fmaxf(v1[c], 0.f)), sg2 = sqrt_fast(fmaxf(v2[c], 0.f));
    const float *e = eps_of(c);
    float sum = 0.f;
    for (int s = lane; s < S; s += 32) {
      float y1 = fmaf(sg1, e[s], mu1);
      const float y2 = fmaf(sg2, e[S + s], mu2);
      if (CONS && !(y1 <= k1 && y2 <= k2)) y1 = kInfeasible;
      sum += hvi(y1, y2);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0 && BOUTE_INB((long long)b * N + c, (long long)gridDim.y * N))
        acq[(size_t)b * N + c] = sum * inv_s;
    if (SEL) sel.add(make_key(sum * inv_s, (unsigned)c), lane);
  }
  }
  if (!SEL) return;
  sel.flush(lane);
  unsigned long long top = sel.top;
  // ---- selection. Block list (tree over the 16 warps); with several blocks
  // per problem, blocks form groups of kSelGroup: the last block of a group to
  // finish merges the group's lists, and the last group of the problem to
  // finish merges the group lists. Counters are set back to zero by the block
  // that consumed them.
  __shared__ unsigned long long lists[16][kWarpK];
  __shared__ int is_last;
  const int G = gridDim.x, Bp = gridDim.y;
  const int ng = (G + kSelGroup - 1) / kSelGroup, grp = blockIdx.x / kSelGroup;
  const int gsize = min(kSelGroup, G - grp * kSelGroup);
  unsigned long long *blk_keys = sel_keys;                           // Bp x G x 32
  unsigned long long *grp_keys = blk_keys + (size_t)Bp * G * kWarpK;  // Bp x ng x 32
  unsigned *grp_cnt = (unsigned *)(grp_keys + (size_t)Bp * ng * kWarpK);  // Bp x ng
  unsigned *prob_cnt = grp_cnt + (size_t)Bp * ng;                         // Bp
  // merges n <= 32 lists at src (32 keys each) with the whole block
  auto merge_lists = [&](const unsigned long long *src, int n) {
    const unsigned long long x0 = warp < n ? __ldcg(src + (size_t)warp * kWarpK + lane) : 0ull;
    const unsigned long long x1 =
        warp + 16 < n ? __ldcg(src + (size_t)(warp + 16) * kWarpK + lane) : 0ull;
    __syncthreads();  // `lists` free again
    return block_merge16(lists, warp_merge_desc(x0, x1, lane), warp, lane);
  };
  // publishes warp 0's list at dst and counts the block in on *cnt; true in
  // every thread of the block that completes the count of `total`
  // (the count is a release: it carries the list and, through the block's
  // barriers, every acquisition value the block wrote)
  auto publish = [&](unsigned long long *dst, unsigned *cnt, int total) {
    if (warp == 0) {
      dst[lane] = top;
      __syncwarp();
      if (lane == 0) is_last = atomic_add_acq_rel_gpu(cnt, 1u) == (unsigned)(total - 1);
    }
    __syncthreads();
    return is_last != 0;
  };
  top = block_merge16(lists, top, warp, lane);
  if (G > 1) {
    if (!publish(blk_keys + ((size_t)b * G + blockIdx.x) * kWarpK, &grp_cnt[(size_t)b * ng + grp],
                 gsize))
      return;
    top = merge_lists(blk_keys + ((size_t)b * G + (size_t)grp * kSelGroup) * kWarpK, gsize);
    if (threadIdx.x == 0) grp_cnt[(size_t)b * ng + grp] = 0u;
    if (ng > 1) {
      if (!publish(grp_keys + ((size_t)b * ng + grp) * kWarpK, &prob_cnt[b], ng)) return;
      top = merge_lists(grp_keys + (size_t)b * ng * kWarpK, ng);
      if (threadIdx.x == 0) prob_cnt[b] = 0u;
    }
  }
  if (warp == 0 && lane < ksel) {
    const unsigned j = key_index(top);
    idx[(size_t)b * ksel + lane] = (long long)j;
    val[(size_t)b * ksel + lane] = __ldcg(acq + (size_t)b * N + j);
  }
}

}  // namespace

namespace {

// Blocks per problem for a grid-stride kernel whose blocks of `threads`
// threads score `per_block` candidates per pass: as many as are resident on
// the device at once, split over the B problems, so that the grid is one wave.
template <class Kern>
unsigned resident_grid_x(Kern kernel, int threads, size_t smem, int B, long long N,
                         int per_block) {
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, threads, smem) != cudaSuccess) {
    cudaGetLastError();
    occ = 1;
  }
  const long long want = (N + per_block - 1) / per_block;
  const long long fit = (long long)num_sms() * std::max(occ, 1) / std::max(1, B);
  return (unsigned)std::max<long long>(1, std::min(want, fit));
}

}  // namespace

int launch_ehvi(const float *mean, const float *var, int B, long long N, const double *front,
                const int *P, int n, const double *ref, const double *cons, float *acq,
                cudaStream_t s) {
  if (N <= 0) return BOUTE_OK;
  const size_t smem = 2 * (size_t)(n + 1) * sizeof(float);
  if (cons) {
    const unsigned gx = resident_grid_x(ehvi2d_kernel<true>, 256, smem, B, N, 256);
    launch_pdl(ehvi2d_kernel<true>, dim3(gx, B), dim3(256), smem, s, mean, var, N, front, P, n,
               ref, cons, acq);
  } else {
    const unsigned gx = resident_grid_x(ehvi2d_kernel<false>, 256, smem, B, N, 256);
    launch_pdl(ehvi2d_kernel<false>, dim3(gx, B), dim3(256), smem, s, mean, var, N, front, P, n,
               ref, cons, acq);
  }
  count_launch();
  return last_launch_status();
}

namespace {

size_t mchvi2_smem(int box_cap) { return ((size_t)box_cap + 4) * sizeof(float4); }

// The dynamic shared-memory limit is set on every launch: the kernels' static
// arrays count against the same 48 KB default as the dynamic part.
template <class Kern>
void configure_smem(Kern kernel, size_t smem) {
  prefer_shared(kernel);
  cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

void mchvi2_configure(int box_cap) {
  const size_t smem = mchvi2_smem(box_cap);
  configure_smem(mchvi2_kernel<true, false>, smem);
  configure_smem(mchvi2_kernel<true, true>, smem);
  configure_smem(mchvi2_kernel<false, false>, smem);
  configure_smem(mchvi2_kernel<false, true>, smem);
}

}  // namespace

// One grid for both variants of the selecting kernel (the scratch is sized by
// it); the grid stride makes any grid correct.
unsigned mchvi2_select_grid_x(int B, long long N, int box_cap) {
  mchvi2_configure(box_cap);
  return resident_grid_x(mchvi2_kernel<true, false>, 512, mchvi2_smem(box_cap), B, N, 16);
}

// Bytes of the selection scratch of launch_mchvi2_select: per problem, one
// list of 32 keys per block and per group of kSelGroup blocks, then one
// counter per group and per problem (zero on entry, zero on exit).
size_t mchvi2_select_scratch_bytes(int B, long long N, int box_cap) {
  const size_t G = mchvi2_select_grid_x(B, N, box_cap), ng = (G + kSelGroup - 1) / kSelGroup;
  return (size_t)B * (G + ng) * kWarpK * sizeof(unsigned long long) +
         (size_t)B * (ng + 1) * sizeof(unsigned);
}

// 2-objective Monte-Carlo HVI with the k <= 32 best candidates selected in the
// same launch; sel: mchvi2_select_scratch_bytes(B, N, box_cap) bytes whose
// counters are zero (they are zero again when the kernel ends).
int launch_mchvi2_select(const float *mean, const float *var, int B, long long N,
                         const float *lower, const float *upper, const int *K, int box_cap,
                         const float *eps, int S, long long eps_stride, const double *cons,
                         float *acq, int k, void *sel, long long *idx, float *val,
                         cudaStream_t s) {
  if (N <= 0 || k < 1 || k > kWarpK || k > N) return BOUTE_ERR_INVALID_ARG;
  const unsigned gx = mchvi2_select_grid_x(B, N, box_cap);
  if (gx > (unsigned)(kSelGroup * kSelGroup)) return BOUTE_ERR_UNSUPPORTED;
  auto *keys = (unsigned long long *)sel;
  if (cons)
    launch_pdl(mchvi2_kernel<true, true>, dim3(gx, B), dim3(16 * 32), mchvi2_smem(box_cap), s,
               mean, var, N, lower, upper, K, box_cap, eps, S, eps_stride, cons, acq, k, keys,
               idx, val);
  else
    launch_pdl(mchvi2_kernel<true, false>, dim3(gx, B), dim3(16 * 32), mchvi2_smem(box_cap), s,
               mean, var, N, lower, upper, K, box_cap, eps, S, eps_stride, cons, acq, k, keys,
               idx, val);
  count_launch();
  return last_launch_status();
}

namespace {

template <bool CONS>
void launch_mchvi2_plain(const float *mean, const float *var, int B, long long N,
                         const float *lower, const float *upper, const int *K, int box_cap,
                         const float *eps, int S, long long eps_stride, const double *cons,
                         float *acq, cudaStream_t s) {
  mchvi2_configure(box_cap);
  const size_t smem = mchvi2_smem(box_cap);
  const unsigned gx = resident_grid_x(mchvi2_kernel<false, CONS>, 512, smem, B, N, 16);
  unsigned long long *nk = nullptr;
  long long *ni = nullptr;
  float *nv = nullptr;
  launch_pdl(mchvi2_kernel<false, CONS>, dim3(gx, B), dim3(16 * 32), smem, s, mean, var, N,
             lower, upper, K, box_cap, eps, S, eps_stride, cons, acq, 0, nk, ni, nv);
}

template <bool CONS>
void launch_mchvi3(const float *mean, const float *var, int B, long long N, const float *lower,
                   const float *upper, const int *K, int box_cap, const float *eps, int S,
                   long long eps_stride, const double *cons, float *acq, cudaStream_t s) {
  const size_t smem = 2 * (size_t)box_cap * 3 * sizeof(float);
  // (the kernel's 16 KB of static staging counts against the same 48 KB
  // default, so the dynamic limit is always set)
  cudaFuncSetAttribute(mchvi_kernel<3, CONS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)smem);
  const unsigned gx = resident_grid_x(mchvi_kernel<3, CONS>, 512, smem, B, N, 16);
  launch_pdl(mchvi_kernel<3, CONS>, dim3(gx, B), dim3(16 * 32), smem, s, mean, var, B, N, lower,
             upper, K, box_cap, eps, S, eps_stride, cons, acq);
}

}  // namespace

int launch_mchvi(const float *mean, const float *var, int B, long long N, int m,
                 const float *lower, const float *upper, const int *K, int box_cap,
                 const float *eps, int S, long long eps_stride, const double *cons, float *acq,
                 cudaStream_t s) {
  if (N <= 0) return BOUTE_OK;
  if (m == 2) {
    if (cons)
      launch_mchvi2_plain<true>(mean, var, B, N, lower, upper, K, box_cap, eps, S, eps_stride,
                                cons, acq, s);
    else
      launch_mchvi2_plain<false>(mean, var, B, N, lower, upper, K, box_cap, eps, S, eps_stride,
                                 cons, acq, s);
  } else if (m == 3) {
    if (cons)
      launch_mchvi3<true>(mean, var, B, N, lower, upper, K, box_cap, eps, S, eps_stride, cons,
                          acq, s);
    else
      launch_mchvi3<false>(mean, var, B, N, lower, upper, K, box_cap, eps, S, eps_stride, cons,
                           acq, s);
  } else {
    return BOUTE_ERR_UNSUPPORTED;
  }
  count_launch();
  return last_launch_status();
}

// ---- Monte-Carlo base normals from a counter-based generator -------------------
// Philox4x64-10 (Salmon et al., SC'11) and the Box-Muller transform, in
// fp64, one thread per block of four samples: samples 4j..4j+3 of candidate
// c, objective t of problem b from counter (j, c, b m + t, 0), key (seed, 0).
namespace {

__device__ __forceinline__ void philox4x64(unsigned long long (&c)[4], unsigned long long k0,
                                           unsigned long long k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const unsigned long long M0 = 0xD2E7470EE14C6C93ull, M1 = 0xCA5A826395121157ull;
    const unsigned long long hi0 = __umul64hi(M0, c[0]), lo0 = M0 * c[0];
    const unsigned long long hi1 = __umul64hi(M1, c[2]), lo1 = M1 * c[2];
    const unsigned long long n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
    c[0] = n0;
    c[1] = lo1;
    c[2] = n2;
    c[3] = lo0;
    k0 += 0x9E3779B97F4A7C15ull;
    k1 += 0xBB67AE8584CAA73Bull;
  }
}

__global__ void normals_kernel(unsigned long long seed, int B, long long N, int m, int S,
                               float *eps) {
  const int J = (S + 3) / 4;
  const long long units = (long long)B * N * m * J;
  for (long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x; u < units;
       u += (long long)gridDim.x * blockDim.x) {
    const int j = (int)(u % J);
    const long long row = u / J;  // (b N + c) m + t
    const int t = (int)(row % m);
    const long long bc = row / m, c = bc % N, b = bc / N;
    unsigned long long w[4] = {(unsigned long long)j, (unsigned long long)c,
                               (unsigned long long)b * m + t, 0ull};
    philox4x64(w, seed, 0ull);
    float z[4];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const double u1 = ((double)(w[2 * q] >> 11) + 0.5) * 0x1p-53;
      const double u2 = ((double)(w[2 * q + 1] >> 11) + 0.5) * 0x1p-53;
      const double rad = sqrt(-2.0 * log(u1));
      double sn, cs;
      sincos(2.0 * M_PI * u2, &sn, &cs);
      z[2 * q] = (float)(rad * cs);
      z[2 * q + 1] = (float)(rad * sn);
    }
    float *e = eps + (size_t)row * S + 4 * j;
    if (4 * j + 4 <= S && ((uintptr_t)e & 15) == 0) {
      *(float4 *)e = make_float4(z[0], z[1], z[2], z[3]);
    } else {
      for (int q = 0; q < 4 && 4 * j + q < S; ++q) e[q] = z[q];
    }
  }
}

}  // namespace

BOUTE_BOUNDS_READER(acq)

int launch_base_normals(unsigned long long seed, int B, long long N, int m, int S, float *eps,
                        cudaStream_t s) {
  const long long units = (long long)B * N * m * ((S + 3) / 4);
  if (units <= 0) return BOUTE_OK;
  const int blocks = (int)std::min<long long>((units + 255) / 256, 32LL * num_sms());
  normals_kernel<<<blocks, 256, 0, s>>>(seed, B, N, m, S, eps);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
