// Fused GP posterior on the 5th-generation tensor cores (sm_103a).
//
// For a tile of 128 candidates and each objective, the Matern-5/2
// cross-covariance K* (128 x n) is built chunk by chunk (32 training points =
// 128 B rows) straight into shared memory in the swizzled K-major operand
// layout, split into tf32 hi/lo parts, and contracted against the prepacked
// operand L^-1 (hi/lo, brought in by bulk TMA copies) with three
// tcgen05.mma kind::tf32 per k-step (hi*hi + hi*lo + lo*hi, fp32 accumulate in
// tensor memory). The variance is s2 - rowsum(V^2), V = K* L^-T, read back
// from tensor memory with tcgen05.ld. The mean K* alpha is a matrix-vector
// product: the threads building K* reduce it on the CUDA cores in fp32 with
// compensated (Kahan) accumulation across chunks, which is more accurate than
// the tensor core's fp32 accumulation and takes no operand column. K* never
// reaches HBM.
//
// Persistent and warp-specialised: each CTA loops over (tile, objective) units.
//   warp 0      bulk-TMA producer of the operand images of L^-1 (B ring)
//   warp 1      tcgen05.mma issuer; owns the 512-column TMEM allocation
//   warps 2-5   epilogue: one TMEM lane quarter each, sum of squares, variance
//   warp 6      bulk-TMA producer of the training-point chunks (side-input ring)
//   warps 7..   K* builders: packed f32x2 distance math, A ring
// Three shared-memory rings with their own depths: A (K* hi/lo, builders ->
// MMA), B (L^-1 hi/lo, TMA -> MMA) and the side input (scaled training points,
// alpha and the objective's parameters, TMA -> builders), so that the builders
// never wait on the operand copies of the MMA; the accumulator is
// double-buffered in TMEM (2 x 256 columns; a pass with a reduction longer
// than 256 takes both buffers, one per half of the reduction) so the
// epilogue of one output pass overlaps the MMAs of the next. Output columns
// beyond 256 are handled in passes; pass p skips the reduction chunks where
// its rows of L^-1 are zero. All waits are bounded (BOUTE_WAIT_NS): a wait
// that gives up records BOUTE_ERR_TIMEOUT and every role stops.
#include <math.h>

#include <algorithm>
#include <type_traits>

#include "internal.h"

namespace boute {

namespace {

constexpr int kEpiWarp0 = 2;  // warps 2-5: epilogue, TMEM lane quarter = warp % 4
constexpr int kEpiWarps = 4;
constexpr int kXtWarp = 6;    // warp 6: side-input producer
constexpr int kBldWarp0 = 7;  // warps 7..: K* builders
constexpr int kMaxA = 4, kMaxB = 4, kMaxX = 8;  // ring depths
constexpr uint32_t kABytes = 32768;             // one A stage: 128 x 32 fp32, hi and lo

// The tensor core's fp32 accumulator truncates after each MMA, so its error
// grows with the number of accumulations into one output. A pass whose
// reduction is longer than 8 chunks (256 training points) accumulates its
// first and second halves in the two TMEM buffers, which the epilogue adds in
// round-to-nearest; returns the chunk count of the first half (kc: no split).
__device__ __forceinline__ int split_chunks(int kc) { return kc > 8 ? (kc + 1) / 2 : kc; }
// builder warps: 16 (8 elements per thread and chunk) when the candidate
// coordinates are short enough to keep in registers, else 8 (16 elements)
template <int DP>
struct Layout {
  static constexpr int kBld = DP <= 16 ? 16 : 8;
  static constexpr int kThreads = 32 * (kBldWarp0 + kBld);
  static constexpr int kCols = 128 / kBld;  // chunk columns per builder thread (8 or 16)
};

struct PostArgs {
  const float *Xc;
  const float *kst;  // precomputed K* (PRE variant), else unused
  float *mean, *var;
  const float *bop, *xt, *s2f;
  int *status;
  long long N;
  int B, m, d, n;
  int tiles_per_problem, tiles_total;
  int sa, sb, sx;              // depths of the A, B and side-input rings
  uint32_t b_bytes, x_bytes;   // one B stage, one side-input entry
  int kern;                    // 1: the composite kernel (prior variance per candidate)
  PostPlan plan;
};

constexpr float kSqrt5 = 2.2360679774997896964f;
constexpr float kSqrt5Log2e = 3.2259641822295610f;  // sqrt(5) / ln(2)
constexpr float kSqrt3 = 1.7320508075688772f;
constexpr float kSqrt3Log2e = 2.4988211106473432f;  // sqrt(3) / ln(2)

// Single hardware instructions (relative error about 2^-22), no range fix-ups:
// arguments here are finite and non-negative (sqrt) or non-positive (ex2).
__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
constexpr float kFiveThirds = 1.6666666666666667f;

// ---- packed fp32 pairs (sm_100+ f32x2 arithmetic) --------------------------------
__device__ __forceinline__ unsigned long long f2_dup(float x) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %1};" : "=l"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ unsigned long long f2_sub(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ unsigned long long f2_fma(unsigned long long a, unsigned long long b,
                                                     unsigned long long c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ void f2_split(unsigned long long v, float &x, float &y) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(v));
}

// 32 lanes x 32 bit, 16 consecutive columns per thread, wait fused.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])::"memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// The composite kernel's per-candidate inputs (Sec. 5.2 "Additive kernels"
// and S5, as Sec. 6 assembles them): the routing features are dimensions
// [0, dtau), the candidate's preference weight w* = exp(beta <s, c*>), the
// outputscales of the weighted deployment term and of the interaction term.
struct CompIn {
  int dtau;
  float ws, s2c, s2x;
};

// The side input's composite-kernel entries within a chunk (the block after
// the scaled coordinates): row 0 the chunk's training-point preference weights
// w_j, row 1 beta * s_k per dimension (zero for routing features); the
// parameter block holds s2_c, s2_x and dtau after the outputscale.
__device__ __forceinline__ const float *chunk_weights(const float *chunk, int DP) {
  return chunk + BOUTE_KCHUNK * DP;
}
__device__ __forceinline__ const float *chunk_pref(const float *chunk, int DP) {
  return chunk + BOUTE_KCHUNK * DP + BOUTE_KCHUNK;
}
__device__ __forceinline__ CompIn chunk_comp(const float *chunk, int DP) {
  const float *pb = chunk + xt_param_offset(DP) + 2 * DP;
  return CompIn{(int)pb[3], 0.f, pb[1], pb[2]};
}

// A candidate's preference weight from its raw coordinates.
template <int DP>
__device__ __forceinline__ float cand_weight(const float (&xr)[DP], const float *bp) {
  float e = 0.f;
#pragma unroll
  for (int k = 0; k < DP; ++k) e = fmaf(bp[k], xr[k], e);
  return expf(e);
}

// The K* values of one builder thread's COLS columns of a 32-point chunk:
// squared scaled distances in packed pairs (candidate x*_k / l_k as a
// duplicated pair, minus the chunk's training coordinates x_k / l_k), then
// k = s2 (1 + sqrt5 r + 5/3 r^2) exp(-sqrt5 r) with exp(-x) = 2^(-x log2 e).
// KERN = 1, the composite kernel: the distances over the routing features
// (r_t) and the deployment features (r_c) are accumulated apart, and
//   k = k52(r_t) (s2 + s2_x k32(r_c)) + s2_c w_j w* k32(r_c),
//   k52(r) = (1 + sqrt5 r + 5/3 r^2) e^(-sqrt5 r), k32(r) = (1 + sqrt3 r) e^(-sqrt3 r).
// Both the fused builders and the stand-alone K* kernel use this, so their
// values are identical.
template <int DP, int COLS, int KERN = 0>
__device__ __forceinline__ void kstar_cols(const unsigned long long (&xs2)[DP], const float *xth,
                                           int g, float s2, float (&kv)[COLS],
                                           const CompIn &ci = CompIn{}) {
  unsigned long long acc2[COLS / 2], accc[COLS / 2];
#pragma unroll
  for (int e = 0; e < COLS / 2; ++e) {
    acc2[e] = 0ull;
    accc[e] = 0ull;
  }
#pragma unroll
  for (int k = 0; k < DP; ++k) {
    // 16-byte loads: two training points' coordinate pairs each
    const ulonglong2 *h4 = (const ulonglong2 *)(xth + k * BOUTE_KCHUNK + COLS * g);
    unsigned long long h2[COLS / 2];
#pragma unroll
    for (int e = 0; e < COLS / 4; ++e) {
      const ulonglong2 v = h4[e];
      h2[2 * e] = v.x;
      h2[2 * e + 1] = v.y;
    }
    if (KERN == 1 && k >= ci.dtau) {  // a deployment feature (uniform branch)
#pragma unroll
      for (int e = 0; e < COLS / 2; ++e) {
        const unsigned long long df = f2_sub(xs2[k], h2[e]);
        accc[e] = f2_fma(df, df, accc[e]);
      }
    } else {
#pragma unroll
      for (int e = 0; e < COLS / 2; ++e) {
        const unsigned long long df = f2_sub(xs2[k], h2[e]);
        acc2[e] = f2_fma(df, df, acc2[e]);
      }
    }
  }
  if (KERN == 1) {
    const float *wj = chunk_weights(xth, DP) + COLS * g;
#pragma unroll
    for (int e = 0; e < COLS / 2; ++e) {
      float r2[2], c2[2];
      f2_split(acc2[e], r2[0], r2[1]);
      f2_split(accc[e], c2[0], c2[1]);
#pragma unroll
      for (int z = 0; z < 2; ++z) {
        const float rr = sqrt_approx(r2[z]);
        const float k52 =
            fmaf(kFiveThirds, r2[z], fmaf(kSqrt5, rr, 1.0f)) * ex2_approx(-kSqrt5Log2e * rr);
        const float rc = sqrt_approx(c2[z]);
        const float k32 = fmaf(kSqrt3, rc, 1.0f) * ex2_approx(-kSqrt3Log2e * rc);
        kv[2 * e + z] = fmaf(k52, fmaf(ci.s2x, k32, s2), ci.s2c * (wj[2 * e + z] * ci.ws) * k32);
      }
    }
    return;
  }
#pragma unroll
  for (int e = 0; e < COLS / 2; ++e) {
    float r2[2];
    f2_split(acc2[e], r2[0], r2[1]);
#pragma unroll
    for (int z = 0; z < 2; ++z) {
      const float rr = sqrt_approx(r2[z]);
      const float sr = kSqrt5 * rr;
      kv[2 * e + z] = s2 * fmaf(kFiveThirds, r2[z], 1.0f + sr) * ex2_approx(-kSqrt5Log2e * rr);
    }
  }
}

// A candidate's scaled coordinates as duplicated pairs, x*_k (1/l_k hi + lo),
// from the objective's parameters (1/l hi [DP], 1/l lo [DP], s2) of a chunk.
template <int DP>
__device__ __forceinline__ void scaled_candidate(const float (&xr)[DP], const float *il,
                                                 unsigned long long (&xs2)[DP]) {
#pragma unroll
  for (int k = 0; k < DP; ++k) xs2[k] = f2_dup(fmaf(xr[k], il[k], xr[k] * il[DP + k]));
}

// Position in a ring of R stages: the stage index and the parity of the
// stage's use count (the mbarrier phase a consumer waits for), advanced
// without integer division.
struct RingPos {
  int idx = 0;
  uint32_t phase = 0;
  __device__ __forceinline__ void advance(int R) {
    if (++idx == R) {
      idx = 0;
      phase ^= 1u;
    }
  }
};

// Bounded wait that also gives up as soon as another role has aborted. The
// waiting thread sleeps in hardware until the phase completes (at most 2 us
// per try), so waiting warps take no issue slots from the K* builders.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity,
                                              volatile int *abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_sleep(bar, parity, 2000)) return true;
    if ((it & 15) == 0) {
      if (*abort) return false;
      if (globaltimer() - t0 > BOUTE_WAIT_NS) {
        *abort = 1;
        return false;
      }
    }
  }
}

// PRE: the K* values come precomputed (kstar_kernel) instead of being built
// here; everything else is the same. KERN: the kernel the builders evaluate
// (0 Matern-5/2, 1 composite; only when !PRE).
template <int DP, bool PRE, int KERN = 0>
__global__ void __launch_bounds__(Layout<DP>::kThreads, 1)
    posterior_kernel(const __grid_constant__ PostArgs a) {
  constexpr int kBldWarps = Layout<DP>::kBld;
  constexpr int COLS = Layout<DP>::kCols;   // columns of a chunk per builder thread
  constexpr int GPR = 32 / COLS;            // column groups per row (threads per row)
  constexpr int RPW = 32 / GPR;             // rows per builder warp
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment (the 128-byte swizzle atom) as an offset from the
  // shared array, so that every access below stays a shared-memory access
  uint8_t *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const PostPlan &pl = a.plan;
  const int n = a.n, m = a.m, d = a.d, SA = a.sa, SB = a.sb, SX = a.sx;
  const int cf = xt_chunk_floats(DP);

  uint8_t *ring_b = sm + (size_t)SA * kABytes;
  uint8_t *ring_x = ring_b + (size_t)SB * a.b_bytes;
  uint64_t *bars = (uint64_t *)(ring_x + (size_t)SX * a.x_bytes);
  uint64_t *a_full = bars, *a_empty = bars + kMaxA;
  uint64_t *b_full = bars + 2 * kMaxA, *b_empty = b_full + kMaxB;
  uint64_t *x_full = b_full + 2 * kMaxB, *x_empty = x_full + kMaxX;
  uint64_t *acc_full = x_full + 2 * kMaxX, *acc_empty = acc_full + 2, *drain = acc_full + 4;
  uint64_t *ahi_full = drain + 1;  // PRE: the K* image of an A stage has landed
  uint32_t *tmem_holder = (uint32_t *)(ahi_full + kMaxA);
  volatile int *abort = (volatile int *)(tmem_holder + 1);

  auto a_hi = [&](int s) { return (float *)(sm + (size_t)s * kABytes); };
  auto a_lo = [&](int s) { return (float *)(sm + (size_t)s * kABytes + 16384); };
  auto b_reg = [&](int s) { return ring_b + (size_t)s * a.b_bytes; };
  auto xt_reg = [&](int j) { return (float *)(ring_x + (size_t)j * a.x_bytes); };

  if (tid == 0) {
    for (int s = 0; s < kMaxA; ++s) {
      mbar_init(&a_full[s], kBldWarps);
      mbar_init(&a_empty[s], 1);
    }
    for (int s = 0; s < kMaxB; ++s) {
      mbar_init(&b_full[s], 1);
      mbar_init(&b_empty[s], 1);
    }
    for (int j = 0; j < kMaxX; ++j) {
      mbar_init(&x_full[j], 1);
      mbar_init(&x_empty[j], kBldWarps);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kEpiWarps);
    }
    mbar_init(drain, 1);
    for (int s = 0; s < kMaxA; ++s) mbar_init(&ahi_full[s], 1);
    *abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_holder, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  pdl_wait();  // the fit's outputs (operand images, side input) are complete

  if (warp == 0 || warp == kXtWarp) {
    // ------------------------------------------------------ producers (B / side input)
    if (lane == 0) {
      const bool is_b = warp == 0;
      const int R = is_b ? SB : SX;
      uint64_t *full = is_b ? b_full : x_full, *empty = is_b ? b_empty : x_empty;
      // PRE: the side-input producer also brings each A stage's K* image (the
      // stage is free once the MMAs that read it have completed)
      const bool with_a = PRE && !is_b;
      uint32_t q = 0;
      RingPos rp, ra;
      int last_q = -1, last_qa = -1;  // last jobs issued
      for (int unit = blockIdx.x; unit < a.tiles_total * m && !*abort; unit += gridDim.x) {
        const int tile = unit / m, t = unit % m;
        const int b = tile / a.tiles_per_problem;
        {
          const int bt = b * m + t;
          for (int p = 0; p < pl.npass && !*abort; ++p) {
            const uint32_t bbytes = (uint32_t)(2 * pl.ncol[p] * 128);
            for (int c = 0; c < pl.kc[p]; ++c, ++q, rp.advance(R), ra.advance(SA)) {
              if (with_a) {
                const int sa = ra.idx;
                if (q >= (uint32_t)SA && !wait_or_abort(&a_empty[sa], ra.phase ^ 1u, abort)) break;
                mbar_arrive_expect_tx(&ahi_full[sa], kABytes / 2);
                bulk_g2s(a_hi(sa),
                         a.kst + ((size_t)unit * pl.nchunk + c) * BOUTE_TILE_M * BOUTE_KCHUNK,
                         kABytes / 2, &ahi_full[sa]);
                last_qa = (int)q;
              }
              const int s = rp.idx;
              if (q >= (uint32_t)R && !wait_or_abort(&empty[s], rp.phase ^ 1u, abort)) break;
              if (is_b) {
                mbar_arrive_expect_tx(&full[s], bbytes);
                bulk_g2s(b_reg(s),
                         a.bop + (size_t)bt * pl.image_floats + pl.off[p] +
                             (size_t)c * 2 * pl.ncol[p] * BOUTE_KCHUNK,
                         bbytes, &full[s]);
              } else {
                mbar_arrive_expect_tx(&full[s], (uint32_t)(cf * 4));
                bulk_g2s(xt_reg(s), a.xt + ((size_t)bt * pl.nchunk + c) * cf, (uint32_t)(cf * 4),
                         &full[s]);
              }
              last_q = (int)q;
            }
          }
        }
      }
      if (*abort) {  // let our copies land before the block exits
        for (int j = std::max(0, last_q - R + 1); j <= last_q; ++j)
          mbar_wait(&full[j % R], (j / R) & 1);
        for (int j = std::max(0, last_qa - SA + 1); j <= last_qa; ++j)
          mbar_wait(&ahi_full[j % SA], (j / SA) & 1);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      uint32_t q = 0, nuse[2] = {0u, 0u};
      int nxt = 0;
      bool issued = false;
      RingPos pa, pb;
      for (int unit = blockIdx.x; unit < a.tiles_total * m && !*abort; unit += gridDim.x) {
        {
          for (int p = 0; p < pl.npass && !*abort; ++p) {
            const int kc = pl.kc[p], h = split_chunks(kc);
            const bool split = h < kc;  // second half of the reduction -> other buffer
            const int A = nxt, Bf = nxt ^ 1;
            if (nuse[A] >= 1 && !wait_or_abort(&acc_empty[A], (nuse[A] - 1) & 1, abort)) break;
            if (split && nuse[Bf] >= 1 &&
                !wait_or_abort(&acc_empty[Bf], (nuse[Bf] - 1) & 1, abort))
              break;
            tc_fence_after();
            const int ncol = pl.ncol[p];
            const uint32_t idesc = idesc_tf32(ncol);
            for (int c = 0; c < kc; ++c, ++q, pa.advance(SA), pb.advance(SB)) {
              const bool second = split && c >= h;
              const uint32_t dtm = tmem + (uint32_t)((second ? Bf : A) * 256);
              const int c0 = second ? h : 0;  // first chunk of this accumulator
              const int sa = pa.idx, sb = pb.idx;
              if (!wait_or_abort(&b_full[sb], pb.phase, abort)) break;
              if (!wait_or_abort(&a_full[sa], pa.phase, abort)) break;
              tc_fence_after();
              const uint32_t sah = smem_u32(a_hi(sa)), sal = smem_u32(a_lo(sa));
              const uint32_t sbh = smem_u32(b_reg(sb)), sbl = sbh + ncol * 128;
#pragma unroll
              for (int ks = 0; ks < 4; ++ks) {
                const uint64_t dah = sdesc_sw128(sah + ks * 32), dal = sdesc_sw128(sal + ks * 32);
                const uint64_t dbh = sdesc_sw128(sbh + ks * 32), dbl = sdesc_sw128(sbl + ks * 32);
                mma_tf32(dtm, dah, dbh, idesc, (c > c0 || ks > 0) ? 1u : 0u);
                mma_tf32(dtm, dah, dbl, idesc, 1u);
                mma_tf32(dtm, dal, dbh, idesc, 1u);
              }
              mma_commit(&a_empty[sa]);
              mma_commit(&b_empty[sb]);
              if (split && c == h - 1) mma_commit(&acc_full[A]);
              issued = true;
            }
            mma_commit(&acc_full[split ? Bf : A]);
            ++nuse[A];
            if (split) ++nuse[Bf];
            else nxt ^= 1;
          }
        }
      }
      if (issued) {  // every MMA of ours has completed before TMEM is released
        mma_commit(drain);
        mbar_wait(drain, 0);
      }
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ---------------------------------------------------------------- epilogue
    const int eq = warp & 3;  // TMEM lane quarter this warp may access
    uint32_t nuse[2] = {0u, 0u};
    int nxt = 0;
    for (int unit = blockIdx.x; unit < a.tiles_total * m && !*abort; unit += gridDim.x) {
      const int tile = unit / m, t = unit % m;
      const int b = tile / a.tiles_per_problem;
      const long long row =
          (long long)(tile % a.tiles_per_problem) * BOUTE_TILE_M + 32 * eq + lane;
      {
        float ss = 0.f;
        for (int p = 0; p < pl.npass; ++p) {
          const int kc = pl.kc[p];
          const bool split = split_chunks(kc) < kc;
          const int A = nxt, Bf = nxt ^ 1;
          if (!wait_or_abort(&acc_full[A], nuse[A] & 1, abort)) break;
          if (split && !wait_or_abort(&acc_full[Bf], nuse[Bf] & 1, abort)) break;
          tc_fence_after();
          const uint32_t lanes = (uint32_t)(32 * eq) << 16;
          const uint32_t ta = tmem + (uint32_t)(A * 256) + lanes;
          const uint32_t tbb = tmem + (uint32_t)(Bf * 256) + lanes;
          for (int cc = 0; cc < pl.ncol[p]; cc += 16) {
            float v[16];
            tmem_ld16(ta + cc, v);
            if (split) {  // V = first half + second half of the reduction
              float w[16];
              tmem_ld16(tbb + cc, w);
#pragma unroll
              for (int e = 0; e < 16; ++e) v[e] += w[e];
            }
#pragma unroll
            for (int e = 0; e < 16; ++e) ss = fmaf(v[e], v[e], ss);  // zero beyond n
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive_count(&acc_empty[A]);
            if (split) mbar_arrive_count(&acc_empty[Bf]);
          }
          ++nuse[A];
          if (split) ++nuse[Bf];
          else nxt ^= 1;
        }
        if (*abort) break;
        if (row < a.N) {
          float prior = a.s2f[b * m + t];
          if (a.kern) {  // composite kernel: k(x, x) = s2 + s2_x + s2_c w(x)^2
            const float *c0 = a.xt + (size_t)(b * m + t) * pl.nchunk * cf;
            const float *bp = chunk_pref(c0, DP), *xrow = a.Xc + ((size_t)b * a.N + row) * d;
            float e = 0.f;
            for (int k = 0; k < d; ++k) e = fmaf(bp[k], xrow[k], e);
            const float w = expf(e);
            prior = fmaf(chunk_comp(c0, DP).s2c * w, w, prior);
          }
          const float vv = prior - ss;
          a.var[((size_t)b * m + t) * a.N + row] = vv > 0.f ? vv : 0.f;
        }
      }
    }
  } else if (warp >= kBldWarp0) {
    // ---------------------------------------------------------------- K* builders
    // thread -> (row r, column group g): COLS consecutive columns of each chunk
    const int bw = warp - kBldWarp0;
    const int r = bw * RPW + lane % RPW, g = lane / RPW;
    uint32_t q = 0;
    RingPos pa, px;
    for (int unit = blockIdx.x; unit < a.tiles_total * m && !*abort; unit += gridDim.x) {
      const int tile = unit / m, t = unit % m;
      const int b = tile / a.tiles_per_problem;
      const long long row = (long long)(tile % a.tiles_per_problem) * BOUTE_TILE_M + r;
      float xr[DP];
      if (!PRE) {
        const float *xrow = a.Xc + ((long long)b * a.N + row) * d;
#pragma unroll
        for (int k = 0; k < DP; ++k) xr[k] = (k < d && row < a.N) ? xrow[k] : 0.f;
      }
      {
        unsigned long long xs2[DP];
        float s2 = 0.f;
        CompIn ci{};
        float mu = 0.f, comp = 0.f;
        for (int p = 0; p < pl.npass && !*abort; ++p) {
          const bool last_pass = p == pl.npass - 1;
          for (int c = 0; c < pl.kc[p]; ++c, ++q, pa.advance(SA), px.advance(SX)) {
            const int s = pa.idx, j = px.idx;
            if (PRE) {
              if (!wait_or_abort(&ahi_full[s], pa.phase, abort)) break;
            } else if (q >= (uint32_t)SA && !wait_or_abort(&a_empty[s], pa.phase ^ 1u, abort)) {
              break;
            }
            if (!wait_or_abort(&x_full[j], px.phase, abort)) break;
            const float *xth = xt_reg(j), *xtl = xth + BOUTE_KCHUNK * DP;  // x hi, x lo
            const float *alp = xtl + BOUTE_KCHUNK * DP;
            if (!PRE && p == 0 && c == 0) {  // new objective: its parameters came with the chunk
              const float *il = xth + xt_param_offset(DP);
              scaled_candidate<DP>(xr, il, xs2);
              s2 = il[2 * DP];
              if (KERN == 1) {
                ci = chunk_comp(xth, DP);
                ci.ws = cand_weight<DP>(xr, chunk_pref(xth, DP));
              }
            }
            float kv[COLS];
            if (PRE) {  // this thread's COLS values of chunk c, from the stage's image
#pragma unroll
              for (int e = 0; e < COLS / 4; ++e) {
                const float4 v = *(const float4 *)(a_hi(s) + sw128_off(r, COLS * g + 4 * e));
                kv[4 * e] = v.x;
                kv[4 * e + 1] = v.y;
                kv[4 * e + 2] = v.z;
                kv[4 * e + 3] = v.w;
              }
            } else {
              kstar_cols<DP, COLS, KERN>(xs2, xth, g, s2, kv, ci);
            }
            const bool full_chunk = (c + 1) * BOUTE_KCHUNK <= n;
            const int jbase = c * BOUTE_KCHUNK + COLS * g;
            const float *alg = alp + COLS * g;
            float mu_part = 0.f;
            float *Ah = a_hi(s), *Al = a_lo(s);
            // kernel values of this thread's COLS columns into the A stage; the
            // last chunk of a ragged n zeroes the columns beyond n
            auto emit = [&](auto ragged) {
#pragma unroll
              for (int g4 = 0; g4 < COLS / 4; ++g4) {
                float vh[4], vl[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const int kk = 4 * g4 + e;
                  float v = kv[kk];
                  if (decltype(ragged)::value) v = (jbase + kk < n) ? v : 0.f;
                  mu_part = fmaf(v, alg[kk], mu_part);
                  // hi keeps the 19 bits the tensor core reads (it truncates an
                  // fp32 operand to tf32); lo = v - hi exactly
                  const float hi = __uint_as_float(__float_as_uint(v) & 0xFFFFE000u);
                  vh[e] = hi;
                  vl[e] = v - hi;
                }
                const int o = sw128_off(r, COLS * g + g4 * 4);
                // (PRE: the stage already holds the full values, which the
                // tensor core reads as their hi parts)
                if (!PRE) *(float4 *)(Ah + o) = make_float4(vh[0], vh[1], vh[2], vh[3]);
                *(float4 *)(Al + o) = make_float4(vl[0], vl[1], vl[2], vl[3]);
              }
            };
            if (full_chunk) emit(std::false_type{});
            else emit(std::true_type{});
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              mbar_arrive_count(&a_full[s]);
              mbar_arrive_count(&x_empty[j]);
            }
            if (last_pass) {  // Kahan: mu += mu_part (the last pass builds every chunk)
              const float yk = mu_part - comp;
              const float tk = mu + yk;
              comp = (tk - mu) - yk;
              mu = tk;
            }
          }
        }
        if (*abort) break;
        float mt = mu - comp;  // sum over the GPR column groups of the row
#pragma unroll
        for (int o = RPW; o < 32; o <<= 1) mt += __shfl_xor_sync(0xffffffffu, mt, o);
        if (g == 0 && row < a.N) a.mean[((size_t)b * m + t) * a.N + row] = mt;
      }
    }
  }

  // ---- teardown -----------------------------------------------------------------
  pdl_trigger();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (tid == 0 && *abort) set_status(a.status, BOUTE_ERR_TIMEOUT);
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, 512);
  }
}

template <int DP>
int launch_dp(const Gp *gp, const float *Xc, const float *kst, long long N, float *mean,
              float *var, cudaStream_t s) {
  PostArgs a;
  a.Xc = Xc;
  a.kst = kst;
  a.mean = mean;
  a.var = var;
  a.bop = gp->bop;
  a.xt = gp->xt;
  a.s2f = gp->s2f;
  a.status = gp->status;
  a.N = N;
  a.B = gp->B;
  a.m = gp->m;
  a.d = gp->d;
  a.n = gp->n;
  a.plan = gp->plan;
  a.kern = gp->kern;
  a.tiles_per_problem = (int)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M);
  a.tiles_total = a.tiles_per_problem * gp->B;
  const int ncolmax = gp->plan.ncol[0];
  a.b_bytes = (uint32_t)(2 * ncolmax * 128);  // a multiple of 1024 (ncol % 16 == 0)
  a.x_bytes = (uint32_t)round_up(xt_chunk_floats(DP) * 4, 16);
  const size_t fixed = 1024 + 512;  // alignment slack, barriers, TMEM address, flag
  const size_t budget = 227 * 1024 - fixed;
  // deepest B ring first (it hides the operand copies), then A, then the side input
  a.sx = kMaxX;
  a.sa = 3;
  a.sb = kMaxB;
  while ((size_t)a.sa * kABytes + (size_t)a.sb * a.b_bytes + (size_t)a.sx * a.x_bytes > budget) {
    if (a.sx > 4) --a.sx;
    else if (a.sb > a.sa) --a.sb;
    else if (a.sa > 2) --a.sa;
    else if (a.sb > 2) --a.sb;
    else return BOUTE_ERR_UNSUPPORTED;
  }
  const size_t smem =
      fixed + (size_t)a.sa * kABytes + (size_t)a.sb * a.b_bytes + (size_t)a.sx * a.x_bytes;
  const int grid = std::max(1, std::min(a.tiles_total * a.m, num_sms()));  // (tile, objective) units
  auto go = [&](auto kern) {
    prefer_shared(kern);
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    launch_pdl(kern, dim3(grid), dim3(Layout<DP>::kThreads), smem, s, a);
  };
  if (kst) go(posterior_kernel<DP, true>);
  else if (gp->kern) go(posterior_kernel<DP, false, 1>);
  else go(posterior_kernel<DP, false>);
  count_launch();
  return last_launch_status();
}

// ---- K* ahead of the fit's results ------------------------------------------------
// One block per (tile, objective) unit, threads laid out as the posterior's
// builders: all n training points' K* values of the tile's 128 candidates, in
// the builders' arithmetic, zero beyond n. Each 32-point chunk is stored as
// the 16 KB image of an A stage (128 rows x 32 fp32, K-major, 128-byte
// swizzle), so that the posterior brings it in with one bulk copy; the tensor
// core reads an fp32 operand truncated to tf32, so the full value serves as
// the hi part. The training points' side input is staged in shared memory.
// It needs the set-up's side input (not the fit's results) and the candidates.
template <int DP, int KERN>
__global__ void __launch_bounds__(Layout<DP>::kBld * 32) kstar_kernel(
    const float *Xc, const float *xt, long long N, int d, int m, int n, int tiles_per_problem,
    int nchunk, float *kst) {
  constexpr int COLS = Layout<DP>::kCols, GPR = 32 / COLS, RPW = 32 / GPR;
  extern __shared__ __align__(16) float xs[];  // nchunk side-input chunks
  const int unit = blockIdx.x, tile = unit / m, t = unit % m, b = tile / tiles_per_problem;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = warp * RPW + lane % RPW, g = lane / RPW;
  const long long row = (long long)(tile % tiles_per_problem) * BOUTE_TILE_M + r;
  const int cf = xt_chunk_floats(DP);  // a multiple of 4
  const float4 *x4 = (const float4 *)(xt + (size_t)(b * m + t) * nchunk * cf);
  for (int e = threadIdx.x; e < nchunk * cf / 4; e += blockDim.x) ((float4 *)xs)[e] = x4[e];
  const float *xrow = Xc + ((long long)b * N + row) * d;
  float xr[DP];
#pragma unroll
  for (int k = 0; k < DP; ++k) xr[k] = (k < d && row < N) ? xrow[k] : 0.f;
  __syncthreads();
  const float *il = xs + xt_param_offset(DP);
  unsigned long long xs2[DP];
  scaled_candidate<DP>(xr, il, xs2);
  const float s2 = il[2 * DP];
  CompIn ci{};
  if (KERN == 1) {
    ci = chunk_comp(xs, DP);
    ci.ws = cand_weight<DP>(xr, chunk_pref(xs, DP));
  }
  for (int c = 0; c < nchunk; ++c) {
    float kv[COLS];
    kstar_cols<DP, COLS, KERN>(xs2, xs + (size_t)c * cf, g, s2, kv, ci);
    const int jbase = c * BOUTE_KCHUNK + COLS * g;
#pragma unroll
    for (int kk = 0; kk < COLS; ++kk) kv[kk] = (jbase + kk < n) ? kv[kk] : 0.f;
    float *img = kst + ((size_t)unit * nchunk + c) * BOUTE_TILE_M * BOUTE_KCHUNK;
#pragma unroll
    for (int g4 = 0; g4 < COLS / 4; ++g4)
      *(float4 *)(img + sw128_off(r, COLS * g + 4 * g4)) =
          make_float4(kv[4 * g4], kv[4 * g4 + 1], kv[4 * g4 + 2], kv[4 * g4 + 3]);
  }
}

template <int DP>
int launch_kstar_dp(const Gp *gp, const float *Xc, long long N, float *kst, cudaStream_t s) {
  const int tpp = (int)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M);
  const int units = tpp * gp->B * gp->m;
  const size_t smem = (size_t)gp->plan.nchunk * xt_chunk_floats(DP) * sizeof(float);
  auto go = [&](auto kern) {
    prefer_shared(kern);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
      return last_launch_status();
    kern<<<units, Layout<DP>::kBld * 32, smem, s>>>(Xc, gp->xt, N, gp->d, gp->m, gp->n, tpp,
                                                    gp->plan.nchunk, kst);
    return (int)BOUTE_OK;
  };
  if (int r = gp->kern ? go(kstar_kernel<DP, 1>) : go(kstar_kernel<DP, 0>)) return r;
  count_launch();
  return last_launch_status();
}

}  // namespace

int launch_posterior(const Gp *gp, const float *Xc, long long N, float *mean, float *var,
                     cudaStream_t s, const float *kst) {
  if (N <= 0) return BOUTE_OK;
  switch (gp->DP) {
    case 8: return launch_dp<8>(gp, Xc, kst, N, mean, var, s);
    case 12: return launch_dp<12>(gp, Xc, kst, N, mean, var, s);
    case 16: return launch_dp<16>(gp, Xc, kst, N, mean, var, s);
    case 24: return launch_dp<24>(gp, Xc, kst, N, mean, var, s);
    case 32: return launch_dp<32>(gp, Xc, kst, N, mean, var, s);
  }
  return BOUTE_ERR_UNSUPPORTED;
}

size_t kstar_floats(const Gp *gp, long long N) {
  const size_t tpp = (size_t)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M);
  return tpp * gp->B * gp->m * gp->plan.nchunk * BOUTE_TILE_M * BOUTE_KCHUNK;
}

int launch_kstar(const Gp *gp, const float *Xc, long long N, float *kst, cudaStream_t s) {
  if (N <= 0) return BOUTE_OK;
  switch (gp->DP) {
    case 8: return launch_kstar_dp<8>(gp, Xc, N, kst, s);
    case 12: return launch_kstar_dp<12>(gp, Xc, N, kst, s);
    case 16: return launch_kstar_dp<16>(gp, Xc, N, kst, s);
    case 24: return launch_kstar_dp<24>(gp, Xc, N, kst, s);
    case 32: return launch_kstar_dp<32>(gp, Xc, N, kst, s);
  }
  return BOUTE_ERR_UNSUPPORTED;
}

}  // namespace boute
