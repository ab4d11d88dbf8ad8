// 2-objective Monte-Carlo hypervolume improvement (Sec. 5.2, "Constrained
// qNEHVI": the expected improvement estimated over base normals), the
// per-candidate arithmetic of the 2-objective acquisition kernel.
//
// Strip decomposition: strips k = 0..K-1 with x-extent [a_k, b_k) (a_0 = -inf,
// a_k = b_{k-1}) and top u_k (u decreasing, u_0 = r2 the largest). For a
// sample y the improvement is
//   sum_k (b_k - max(a_k, y1))^+ (u_k - y2)^+
//     = (b_0 - y1)^+ (u_0 - y2)^+ + H sum_{k>=1} D_k sat((b_k - y1) / D_k) sat((u_k - y2) / H)
// with D_k = b_k - a_k, because (b_k - max(a_k, y1))^+ is (b_k - y1) clamped
// to [0, D_k], and with H = u_0 - min y2 >= u_k - y2 over the samples a thread
// holds, so that (u_k - y2)^+ = H sat((u_k - y2) / H). Per strip and sample:
// two saturating FMAs and one FMA.
#pragma once

#include <cuda_runtime.h>

namespace boute {

__device__ __forceinline__ float fma_sat(float a, float b, float c) {
  float d;
  asm("fma.rn.sat.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ float sqrt_fast(float x) {
  float y;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcp_fast(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Strips of problem b into shared memory, written by `nthr` threads (thread
// index `t`): [0] = (b_0, u_0, 0, 0), [k >= 1] = (b_k / D_k, 1 / D_k, u_k, D_k)
// (zero width: (0, 0, u_k, 0)), then at most one zero strip so that Kp = 1 + an
// even number (it adds exactly nothing). lower / upper: B x box_cap x 2.
// Returns K.
__device__ __forceinline__ int mc2_load_strips(float4 *strips4, const float *lower,
                                               const float *upper, const int *Kc, int b,
                                               int box_cap, int t, int nthr) {
  const int K = BOUTE_INB(Kc[b], box_cap + 1) ? Kc[b] : 0;
  const int Kp = K > 0 ? 1 + (K & ~1) : 0;
  for (int i = t; i < Kp; i += nthr) {
    if (i >= K) {
      strips4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      continue;
    }
    const size_t o = ((size_t)b * box_cap + i) * 2;
    const float ai = lower[o], bi = upper[o], ui = upper[o + 1];
    if (i == 0) {
      strips4[0] = make_float4(bi, ui, 0.f, 0.f);
    } else {
      const float D = bi - ai;
      strips4[i] = D > 0.f ? make_float4(bi / D, 1.f / D, ui, D) : make_float4(0.f, 0.f, ui, 0.f);
    }
  }
  return K;
}

__device__ __forceinline__ int mc2_padded(int K) { return K > 0 ? 1 + (K & ~1) : 0; }

// A sample that violates a constraint contributes nothing (Sec. 5.2,
// constrained qNEHVI: HVI times the feasibility indicator): its first
// coordinate is moved beyond every strip, which makes every width term zero.
constexpr float kInfeasible = 3.0e38f;

// One lane's share of the improvement sum of a candidate, S = 128: the lane's
// four samples per objective (c1, c2: base normals), posterior mean mu and
// variance pv per objective. t0 = strips4[0] (zero when K = 0), u0 = t0.y.
// CONS: samples count only if y_1 <= k1 and y_2 <= k2 (thresholds on the
// minimised objectives). The caller adds the 32 lanes' shares and divides by S.
template <bool CONS = false>
__device__ __forceinline__ float mc2_lane_sum(const float4 *strips4, int K, int Kp, float4 t0,
                                              float4 c1, float4 c2, float mu1, float mu2,
                                              float pv1, float pv2, float k1 = 0.f,
                                              float k2 = 0.f) {
  const float u0 = t0.y;
  const float sg1 = sqrt_fast(fmaxf(pv1, 0.f)), sg2 = sqrt_fast(fmaxf(pv2, 0.f));
  const float y1c[4] = {fmaf(sg1, c1.x, mu1), fmaf(sg1, c1.y, mu1), fmaf(sg1, c1.z, mu1),
                        fmaf(sg1, c1.w, mu1)};
  const float y2[4] = {fmaf(sg2, c2.x, mu2), fmaf(sg2, c2.y, mu2), fmaf(sg2, c2.z, mu2),
                       fmaf(sg2, c2.w, mu2)};
  float y1[4] = {y1c[0], y1c[1], y1c[2], y1c[3]};
  if (CONS) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (!(y1c[j] <= k1 && y2[j] <= k2)) y1[j] = kInfeasible;
  }
  // per lane: H = u_0 - (its lowest y2) bounds every height of its samples
  const float lo2 = fminf(fminf(y2[0], y2[1]), fminf(y2[2], y2[3]));
  const float H = u0 - lo2;
  float sum = 0.f;
  if (K > 0) {
#pragma unroll
    for (int j = 0; j < 4; ++j) sum += fmaxf(t0.x - y1[j], 0.f) * fmaxf(t0.y - y2[j], 0.f);
    const float iH = H > 0.f ? rcp_fast(H) : 0.f;  // H <= 0: every sample dominated
    // height of strip k for sample j: sat(u_k / H - y2_j / H)
    const float ny2[4] = {-y2[0] * iH, -y2[1] * iH, -y2[2] * iH, -y2[3] * iH};
    float acc = 0.f;
    auto strip = [&](const float4 t) {
      float tk = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        tk = fmaf(fma_sat(-y1[j], t.y, t.x), fma_sat(t.z, iH, ny2[j]), tk);
      acc = fmaf(t.w, tk, acc);
    };
    int k = 1;
#pragma unroll 1
    for (; k + 3 < Kp; k += 4) {
#pragma unroll
      for (int q = 0; q < 4; ++q) strip(strips4[k + q]);
    }
    if (k < Kp) {  // Kp - 1 is even: two strips remain
      strip(strips4[k]);
      strip(strips4[k + 1]);
    }
    sum = fmaf(fmaxf(H, 0.f), acc, sum);
  }
  return sum;
}

// The warp's total of the lanes' shares (every lane receives it).
__device__ __forceinline__ float mc2_warp_total(float sum) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  return sum;
}

}  // namespace boute
