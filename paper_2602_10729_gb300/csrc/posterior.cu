// Fused GP posterior on the 5th-generation tensor cores (sm_103a).
//
// For a tile of 128 candidates and each objective, the Matern-5/2
// cross-covariance K* (128 x n) is built chunk by chunk (32 training points =
// 128 B rows) straight into shared memory in the swizzled K-major operand
// layout, split into tf32 hi/lo parts, and contracted against the prepacked
// operand L^-1 (hi/lo, brought in by bulk TMA copies) with three
// tcgen05.mma kind::tf32 per k-step (hi*hi + hi*lo + lo*hi, fp32 accumulate in
// tensor memory). The epilogue reads the 128 x ncol accumulator back with
// tcgen05.ld and reduces it to the variance s2 - rowsum(V^2). The mean K* alpha
// is a matrix-vector product: the threads building K* reduce it on the CUDA
// cores in fp32 with compensated (Kahan) accumulation across chunks, which is
// more accurate than the tensor core's fp32 accumulation and takes no
// operand column. K* never reaches HBM.
//
// Pipeline: two shared-memory stages. While the tensor core runs chunk q-1,
// the 256 threads build chunk q and the TMA engine fetches chunk q+1's
// operand image. Output columns beyond 256 are handled in passes (TMEM holds
// the 128 x 256 fp32 accumulator); pass p skips the reduction chunks where its
// rows of L^-1 are zero.
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace boute {

namespace {

struct PostArgs {
  const float *Xc;
  float *mean, *var;
  const float *bop, *xt, *invls, *s2f;
  int *status;
  long long N;
  int m, d, n;
  uint32_t stage_bytes;
  PostPlan plan;
};

constexpr float kSqrt5 = 2.2360679774997896964f;
constexpr float kFiveThirds = 1.6666666666666667f;

template <int DP>
__global__ void __launch_bounds__(256, 1) posterior_kernel(const __grid_constant__ PostArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *sm = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int row = tid & 127, half = tid >> 7;
  const int b = blockIdx.y;
  const long long tile0 = (long long)blockIdx.x * BOUTE_TILE_M;
  const PostPlan &pl = a.plan;
  const int n = a.n, m = a.m, d = a.d;

  uint64_t *bars = (uint64_t *)(sm + 2 * a.stage_bytes);
  uint64_t *full = bars, *empty = bars + 2, *accb = bars + 4, *xbar = bars + 5,
           *drain = bars + 6;
  uint32_t *tmem_holder = (uint32_t *)(bars + 7);
  float *red_ss = (float *)(bars + 8);  // [2][128]
  float *red_mu = red_ss + 256;         // [2][128]
  __shared__ int s_abort;

  auto stage = [&](int s) { return sm + (size_t)s * a.stage_bytes; };
  auto a_hi = [&](int s) { return (float *)stage(s); };
  auto a_lo = [&](int s) { return (float *)(stage(s) + 16384); };
  auto b_reg = [&](int s) { return stage(s) + 32768; };
  const int ncolmax = pl.ncol[0];
  auto xt_reg = [&](int s) { return (float *)(stage(s) + 32768 + 2 * ncolmax * 128); };
  const int cf = xt_chunk_floats(DP);

  if (tid == 0) {
    for (int i = 0; i < 7; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
    s_abort = 0;
  }
  if (warp == 0) {
    tmem_alloc(tmem_holder, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  // ---- candidate tile -> registers (raw coordinates) -----------------------
  const long long rows_here = std::min<long long>(BOUTE_TILE_M, a.N - tile0);
  const float *xsrc = a.Xc + ((long long)b * a.N + tile0) * d;
  const uint32_t xbytes = (uint32_t)(BOUTE_TILE_M * d * 4);
  const bool x_tma = rows_here == BOUTE_TILE_M && ((uintptr_t)xsrc & 15) == 0 && (xbytes & 15) == 0;
  float xr[DP];
  if (x_tma) {
    // staged through stage 1's A region, which is first written by chunk 1
    if (tid == 0) {
      mbar_arrive_expect_tx(xbar, xbytes);
      bulk_g2s(a_hi(1), xsrc, xbytes, xbar);
    }
    if (!mbar_wait(xbar, 0)) s_abort = 1;
    const float *xs = a_hi(1) + row * d;
#pragma unroll
    for (int t = 0; t < DP; ++t) xr[t] = t < d ? xs[t] : 0.f;
  } else {
#pragma unroll
    for (int t = 0; t < DP; ++t) xr[t] = (t < d && row < rows_here) ? xsrc[(long long)row * d + t] : 0.f;
  }
  __syncthreads();

  // ---- job sequence: objective t, pass p, chunk c -------------------------
  int total = 0;
  for (int p = 0; p < pl.npass; ++p) total += pl.kc[p];
  total *= m;

  auto issue = [&](int t, int p, int c, int s) {
    const int bt = b * m + t;
    const uint32_t bbytes = (uint32_t)(2 * pl.ncol[p] * 128);
    const uint32_t xtb = (uint32_t)(cf * 4);
    mbar_arrive_expect_tx(&full[s], bbytes + xtb);
    bulk_g2s(b_reg(s),
             a.bop + (size_t)bt * pl.image_floats + pl.off[p] +
                 (size_t)c * 2 * pl.ncol[p] * BOUTE_KCHUNK,
             bbytes, &full[s]);
    bulk_g2s(xt_reg(s), a.xt + ((size_t)bt * pl.nchunk + c) * cf, xtb, &full[s]);
  };
  auto next_job = [&](int &t, int &p, int &c) {
    if (++c == pl.kc[p]) {
      c = 0;
      if (++p == pl.npass) {
        p = 0;
        ++t;
      }
    }
  };

  int pend_q[2] = {-1, -1};  // thread 0: job whose TMA is issued but not yet consumed
  if (tid == 0 && !s_abort && total > 0) {
    issue(0, 0, 0, 0);
    pend_q[0] = 0;
  }
  int nt = 0, np = 0, nc = 0;  // job q+1
  next_job(nt, np, nc);
  int t = 0, p = 0, c = 0;
  int pass_count = 0;
  float xs[DP];
  float s2 = 0.f, ss_acc = 0.f, mu_acc = 0.f, mu_comp = 0.f;
  bool mma_issued = false;

  for (int q = 0; q < total; ++q) {
    const int s = q & 1;
    // (1) prefetch job q+1 into the other stage once the MMAs of job q-1 are done
    if (tid == 0 && q + 1 < total && !s_abort) {
      const int s1 = (q + 1) & 1;
      bool ok = true;
      if (q + 1 >= 2) ok = mbar_wait(&empty[s1], (((q + 1) >> 1) - 1) & 1);
      if (ok) {
        issue(nt, np, nc, s1);
        pend_q[s1] = q + 1;
      } else {
        s_abort = 1;
      }
    }
    // (2) operands of job q landed
    if (!mbar_wait(&full[s], (q >> 1) & 1)) s_abort = 1;
    if (tid == 0) pend_q[s] = -1;
    // (3) new objective: scaled candidate coordinates
    if (p == 0 && c == 0) {
      const int bt = b * m + t;
      const float *il = a.invls + (size_t)bt * 2 * DP;
#pragma unroll
      for (int k = 0; k < DP; ++k) xs[k] = fmaf(xr[k], il[k], xr[k] * il[DP + k]);
      s2 = a.s2f[bt];
      ss_acc = 0.f;
      mu_acc = 0.f;
      mu_comp = 0.f;
    }
    // build K* chunk c: this thread's row, 16 columns [16*half, 16*half+16)
    {
      const float *xth = xt_reg(s), *xtl = xth + BOUTE_KCHUNK * DP;
      const float *alp = xth + 2 * BOUTE_KCHUNK * DP;
      float *Ah = a_hi(s), *Al = a_lo(s);
      const int jbase = c * BOUTE_KCHUNK;
      float mu_part = 0.f;
#pragma unroll
      for (int g4 = 0; g4 < 4; ++g4) {
        float vh[4], vl[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int kk = half * 16 + g4 * 4 + e;
          const float4 *ph = (const float4 *)(xth + kk * DP);
          const float4 *plo = (const float4 *)(xtl + kk * DP);
          float acc = 0.f;
#pragma unroll
          for (int q4 = 0; q4 < DP / 4; ++q4) {
            const float4 h4 = ph[q4], l4 = plo[q4];
            float df;
            df = (xs[4 * q4 + 0] - h4.x) - l4.x; acc = fmaf(df, df, acc);
            df = (xs[4 * q4 + 1] - h4.y) - l4.y; acc = fmaf(df, df, acc);
            df = (xs[4 * q4 + 2] - h4.z) - l4.z; acc = fmaf(df, df, acc);
            df = (xs[4 * q4 + 3] - h4.w) - l4.w; acc = fmaf(df, df, acc);
          }
          const float r = sqrtf(acc);
          const float sr = kSqrt5 * r;
          float kv = s2 * fmaf(kFiveThirds, acc, 1.0f + sr) * expf(-sr);
          kv = (jbase + kk < n) ? kv : 0.f;
          mu_part = fmaf(kv, alp[kk], mu_part);  // used in the last pass only
          const float hi = tf32_rna(kv);
          vh[e] = hi;
          vl[e] = kv - hi;
        }
        const int o = sw128_off(row, half * 16 + g4 * 4);
        *(float4 *)(Ah + o) = make_float4(vh[0], vh[1], vh[2], vh[3]);
        *(float4 *)(Al + o) = make_float4(vl[0], vl[1], vl[2], vl[3]);
      }
      // Kahan: mu_acc += mu_part, once per chunk: the last pass builds every
      // chunk, earlier passes rebuild a prefix of them
      if (p == pl.npass - 1) {
        const float yk = mu_part - mu_comp;
        const float tk = mu_acc + yk;
        mu_comp = (tk - mu_acc) - yk;
        mu_acc = tk;
      }
    }
    // (4) publish the chunk to the tensor core
    fence_proxy_async_smem();
    __syncthreads();
    if (s_abort) break;
    const int ncol = pl.ncol[p];
    const bool last_chunk = c == pl.kc[p] - 1;
    // (5) one thread issues 4 k-steps x 3 MMAs
    if (tid == 0) {
      tc_fence_after();
      const uint32_t idesc = idesc_tf32(ncol);
      const uint32_t sah = smem_u32(a_hi(s)), sal = smem_u32(a_lo(s));
      const uint32_t sbh = smem_u32(b_reg(s)), sbl = sbh + ncol * 128;
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        const uint64_t dah = sdesc_sw128(sah + ks * 32), dal = sdesc_sw128(sal + ks * 32);
        const uint64_t dbh = sdesc_sw128(sbh + ks * 32), dbl = sdesc_sw128(sbl + ks * 32);
        mma_tf32(tmem, dah, dbh, idesc, (c > 0 || ks > 0) ? 1u : 0u);
        mma_tf32(tmem, dah, dbl, idesc, 1u);
        mma_tf32(tmem, dal, dbh, idesc, 1u);
      }
      mma_commit(&empty[s]);
      if (last_chunk) mma_commit(accb);
      mma_issued = true;
    }
    // (6) end of pass: drain the accumulator
    if (last_chunk) {
      if (!mbar_wait(accb, pass_count & 1)) s_abort = 1;
      __syncthreads();  // a uniform abort decision before the warp-collective loads
      if (s_abort) break;
      tc_fence_after();
      const int gq = warp & 3, hsel = warp >> 2;
      const int hcols = ncol >> 1;
      const uint32_t tbase = tmem + ((uint32_t)(32 * gq) << 16) + (uint32_t)(hsel * hcols);
      for (int cc = 0; cc < hcols; cc += 8) {
        float v[8];
        tmem_ld8(tbase + cc, v);
#pragma unroll
        for (int e = 0; e < 8; ++e) ss_acc = fmaf(v[e], v[e], ss_acc);  // zero beyond n
      }
      tc_fence_before();
      __syncthreads();
      ++pass_count;
      if (p == pl.npass - 1) {  // objective complete
        const int r2 = 32 * gq + lane;
        red_ss[hsel * 128 + r2] = ss_acc;
        red_mu[half * 128 + row] = mu_acc - mu_comp;
        __syncthreads();
        if (half == 0) {
          const long long gr = tile0 + row;
          if (gr < a.N) {
            const size_t o = ((size_t)b * m + t) * a.N + gr;
            const float vv = s2 - (red_ss[row] + red_ss[128 + row]);
            a.mean[o] = red_mu[row] + red_mu[128 + row];
            a.var[o] = vv > 0.f ? vv : 0.f;
          }
        }
        __syncthreads();
      }
    }
    t = nt; p = np; c = nc;
    next_job(nt, np, nc);
  }

  // ---- teardown: nothing of ours may still be in flight ---------------------
  if (tid == 0) {
    if (s_abort) set_status(a.status, BOUTE_ERR_TIMEOUT);
    if (mma_issued) {
      mma_commit(drain);
      mbar_wait(drain, 0);
    }
    for (int s = 0; s < 2; ++s)
      if (pend_q[s] >= 0) mbar_wait(&full[s], (pend_q[s] >> 1) & 1);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

template <int DP>
int launch_dp(const Gp *gp, const float *Xc, long long N, float *mean, float *var,
              cudaStream_t s) {
  PostArgs a;
  a.Xc = Xc;
  a.mean = mean;
  a.var = var;
  a.bop = gp->bop;
  a.xt = gp->xt;
  a.invls = gp->invls;
  a.s2f = gp->s2f;
  a.status = gp->status;
  a.N = N;
  a.m = gp->m;
  a.d = gp->d;
  a.n = gp->n;
  a.plan = gp->plan;
  const int ncolmax = gp->plan.ncol[0];
  a.stage_bytes = (uint32_t)round_up(32768 + 2 * ncolmax * 128 + xt_chunk_floats(DP) * 4, 1024);
  const size_t smem = 1024 + 2 * (size_t)a.stage_bytes + 8 * 8 + 2 * 256 * 4;
  cudaFuncSetAttribute(posterior_kernel<DP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)smem);
  dim3 grid((unsigned)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M), gp->B);
  posterior_kernel<DP><<<grid, 256, smem, s>>>(a);
  count_launch();
  return last_launch_status();
}

}  // namespace

int launch_posterior(const Gp *gp, const float *Xc, long long N, float *mean, float *var,
                     cudaStream_t s) {
  if (N <= 0) return BOUTE_OK;
  switch (gp->DP) {
    case 8: return launch_dp<8>(gp, Xc, N, mean, var, s);
    case 12: return launch_dp<12>(gp, Xc, N, mean, var, s);
    case 16: return launch_dp<16>(gp, Xc, N, mean, var, s);
    case 24: return launch_dp<24>(gp, Xc, N, mean, var, s);
    case 32: return launch_dp<32>(gp, Xc, N, mean, var, s);
  }
  return BOUTE_ERR_UNSUPPORTED;
}

}  // namespace boute
