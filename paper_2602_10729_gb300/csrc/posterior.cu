// Fused GP posterior on the 5th-generation tensor cores (sm_103a).
//
// For a tile of 128 candidates and each objective, the Matern-5/2
// cross-covariance K* (128 x n) is built chunk by chunk (64 training points =
// one 128-byte row of fp16 per candidate) straight into shared memory in the
// swizzled K-major operand layout, split into fp16 hi/lo parts, and
// contracted against the prepacked operand W = L^-1 (fp16 hi/lo, brought in by
// bulk TMA copies) with three tcgen05.mma kind::f16 per k-step (hi*hi + hi*lo
// + lo*hi, fp32 accumulate in tensor memory): 22 significant bits per operand
// at twice the tensor rate of tf32. Both operands are scaled by powers of two
// into fp16's normal range (K* by 2^e_r from its bound, W by 2^e_W from
// ||L^-1|| <= 1/sigma_n), which the epilogue divides out exactly. The
// variance is s2 - rowsum(V^2), V = K* W^T, read back from tensor memory with
// tcgen05.ld. The mean K* alpha is a matrix-vector product: the threads
// building K* reduce it on the CUDA cores from the fp32 values, with
// compensated (Kahan) accumulation across chunks, which is more accurate than
// the tensor core's fp32 accumulation and takes no operand column. K* never
// reaches HBM.
//
// Output columns come in blocks of 128, one per tensor-memory slot (4 slots
// of 128 columns, assigned round-robin over the blocks a CTA processes, so the
// epilogue of one block overlaps the MMAs of later ones). Up to four blocks
// form a group that shares each K* chunk: the chunk is built once and feeds
// every block of the group whose rows of W are not zero there (block q needs
// chunks [0, kc[q])). With n <= 512 every chunk is built once per tile.
//
// Persistent and warp-specialised: each CTA loops over (tile, objective) units.
//   warp 0      bulk-TMA producer of the operand images of W (B ring)
//   warp 1      tcgen05.mma issuer; owns the 512-column TMEM allocation
//   warps 2-5   epilogue: one TMEM lane quarter each, sum of squares, variance
//   warp 6      bulk-TMA producer of the training-point chunks (side-input ring)
//               and, with K* precomputed, of its fp32 images (staging ring)
//   warps 7..   K* builders: packed f32x2 distance math, A ring
// All waits are bounded (BOUTE_WAIT_NS): a wait that gives up records
// BOUTE_ERR_TIMEOUT and every role stops.
#include <math.h>

#include <algorithm>
#include <type_traits>

#include "internal.h"

namespace boute {

namespace {

constexpr int kEpiWarp0 = 2;  // warps 2-5: epilogue (variance, mean), TMEM lane quarter = warp % 4
constexpr int kEpiWarps = 4;
constexpr int kXtWarp = 6;     // warp 6: side-input producer
constexpr int kCacheWarp = 7;  // warp 7 (8 builder warps): cached K* chunks into their A stages
constexpr int kMaxA = 4, kMaxB = 6, kMaxX = 8;  // ring depths
constexpr int kSlots = 4;                       // TMEM accumulator slots of 128 columns
constexpr int kGroup = 4;                       // blocks sharing one K* chunk
constexpr uint32_t kAPartBytes = BOUTE_TILE_M * BOUTE_ACHUNK * 2;   // one fp16 part: 16 KB
constexpr uint32_t kABytes = 2 * kAPartBytes;                       // hi and lo
constexpr uint32_t kStageBytes = BOUTE_TILE_M * BOUTE_ACHUNK * 4;   // fp32 K* image: 32 KB

// builder warps: 16 (8 columns of each 32-point half per thread) when the
// candidate coordinates are short enough to keep in registers, else 8 (16
// columns of one row, or 8 columns of two rows: kstar_pair)
template <int DP>
struct Layout {
  static constexpr int kBld = DP <= 16 ? 16 : 8;
  // with 8 builder warps the cached K* chunks have a warp of their own (warp
  // 7); with 16 the side-input producer brings them (a 25th warp would cost
  // the builders registers), and the builders start at warp 7
  static constexpr bool kSepCache = kBld == 8;
  static constexpr int kBldWarp0 = kSepCache ? 8 : 7;
  static constexpr int kThreads = 32 * (kBldWarp0 + kBld);
  static constexpr int kCols = 128 / kBld;  // columns of a 32-point half per builder thread
};

struct PostArgs {
  const float *Xc;
  const float *kst;  // precomputed K* (PRE variant), else unused
  float *mean, *var;
  // in-sample draws (plan.S_in > 0): the shifts l^T z_s, B x m x S_in x N;
  // var then receives the conditional variance
  float *shift;
  const uint16_t *bop;
  const float *xt, *s2f;
  int *status;
  long long N;
  int B, m, d, n;
  int tiles_per_problem, tiles_total;
  int sa, sb, sx;              // depths of the A (and staging), B and side-input rings
  uint32_t b_bytes, x_bytes;   // one B stage, one side-input entry
  int kern;                    // 1: the composite kernel (prior variance per candidate)
  // K* chunks built by one group and needed again by later groups: kept as
  // their fp16 A-stage images in this CTA's slots of kcache (ncache chunks
  // per CTA, 0 = rebuilt instead)
  uint16_t *kcache;
  int ncache;
  PostPlan plan;
};

// Word offset, inside a [128 x 64] fp32 K* image (PRE), of element (row, kk):
// 16-byte groups permuted by XOR with (row mod 16), so that a builder warp's
// rows read distinct banks.
__host__ __device__ __forceinline__ int st_off32(int row, int kk) {
  return row * 64 + ((((kk >> 2) ^ (row & 15))) << 2) + (kk & 3);
}


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
// In the scaled distance r' = sqrt5 r / ln 2 (sqrt3 r / ln 2 for Matern-3/2):
// sqrt5 r = ln2 r', 5/3 r^2 = (ln2)^2 / 3 r'^2, exp(-sqrt5 r) = 2^(-r').
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLn2Sq3 = 0.16015100463940046f;  // (ln 2)^2 / 3

// Compensated (Kahan) accumulation of packed pairs: s + c carries the sum
// of the terms with the rounding error of every addition.
struct Kahan2 {
  unsigned long long s = 0ull, c = 0ull;
  __device__ __forceinline__ void add(unsigned long long x) {
    const unsigned long long y = f2_sub(x, c);
    const unsigned long long t = f2_add(s, y);
    c = f2_sub(f2_sub(t, s), y);
    s = t;
  }
};
// Error-free sum of two floats (Knuth).
__device__ __forceinline__ void two_sum_f(float a, float b, float &s, float &e) {
  s = a + b;
  const float bb = s - a;
  e = (a - (s - bb)) + (b - bb);
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
// duplicated pair, minus the chunk's training coordinates x_k / l_k, both
// times the side input's coordinate scale), then
// k = s2 (1 + sqrt5 r + 5/3 r^2) exp(-sqrt5 r) = s2 (1 + ln2 r' + ln2^2/3 r'^2) 2^(-r').
// KERN = 1, the composite kernel: the distances over the routing features
// (r_t) and the deployment features (r_c) are accumulated apart, and
//   k = k52(r_t) (s2 + s2_x k32(r_c)) + s2_c w_j w* k32(r_c),
//   k52(r) = (1 + sqrt5 r + 5/3 r^2) e^(-sqrt5 r), k32(r) = (1 + sqrt3 r) e^(-sqrt3 r),
// each in its own scaled distance (the deployment features carry sqrt3 / ln 2).
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
        const float k52 = fmaf(kLn2Sq3, r2[z], fmaf(kLn2, rr, 1.0f)) * ex2_approx(-rr);
        const float rc = sqrt_approx(c2[z]);
        const float k32 = fmaf(kLn2, rc, 1.0f) * ex2_approx(-rc);
        kv[2 * e + z] = fmaf(k52, fmaf(ci.s2x, k32, s2), ci.s2c * (wj[2 * e + z] * ci.ws) * k32);
      }
    }
    return;
  }
  // packed pairs: k = (s2 + s2 ln2 r' + s2 ln2^2/3 r'^2) 2^(-r'); the exponent
  // is the scaled distance itself, so the exponential is as accurate as ex2
  const unsigned long long c0 = f2_dup(s2), c1 = f2_dup(s2 * kLn2), c2 = f2_dup(s2 * kLn2Sq3);
#pragma unroll
  for (int e = 0; e < COLS / 2; ++e) {
    float ra, rb;
    f2_split(acc2[e], ra, rb);
    const float r0 = sqrt_approx(ra), r1 = sqrt_approx(rb);
    const unsigned long long ex = f2_pack(ex2_approx(-r0), ex2_approx(-r1));
    const unsigned long long t = f2_fma(acc2[e], c2, f2_fma(f2_pack(r0, r1), c1, c0));
    f2_split(f2_mul(t, ex), kv[2 * e], kv[2 * e + 1]);
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

// Two candidates' scaled coordinates as (row 0, row 1) pairs.
template <int DP>
__device__ __forceinline__ void scaled_pair(const float (&x0)[DP], const float (&x1)[DP],
                                            const float *il, unsigned long long (&xs2)[DP]) {
#pragma unroll
  for (int k = 0; k < DP; ++k)
    xs2[k] = f2_pack(fmaf(x0[k], il[k], x0[k] * il[DP + k]), fmaf(x1[k], il[k], x1[k] * il[DP + k]));
}

// kstar_cols for a pair of candidate rows (Matern-5/2): C columns of a 32-point
// chunk, each value a (row 0, row 1) pair; every training coordinate is loaded
// once for the two rows and duplicated in registers. Per entry the same
// operations in the same order as kstar_cols, so the values are identical.
template <int DP, int C>
__device__ __forceinline__ void kstar_pair(const unsigned long long (&xs2)[DP], const float *xth,
                                           int g, float s2, unsigned long long (&kv)[C]) {
  unsigned long long acc[C];
#pragma unroll
  for (int e = 0; e < C; ++e) acc[e] = 0ull;
#pragma unroll
  for (int k = 0; k < DP; ++k) {
    const float4 *h4 = (const float4 *)(xth + k * BOUTE_KCHUNK + C * g);
    float h[C];
#pragma unroll
    for (int e = 0; e < C / 4; ++e) {
      const float4 v = h4[e];
      h[4 * e] = v.x;
      h[4 * e + 1] = v.y;
      h[4 * e + 2] = v.z;
      h[4 * e + 3] = v.w;
    }
#pragma unroll
    for (int e = 0; e < C; ++e) {
      const unsigned long long df = f2_sub(xs2[k], f2_dup(h[e]));
      acc[e] = f2_fma(df, df, acc[e]);
    }
  }
  const unsigned long long c0 = f2_dup(s2), c1 = f2_dup(s2 * kLn2), c2 = f2_dup(s2 * kLn2Sq3);
#pragma unroll
  for (int e = 0; e < C; ++e) {
    float ra, rb;
    f2_split(acc[e], ra, rb);
    const float r0 = sqrt_approx(ra), r1 = sqrt_approx(rb);
    const unsigned long long ex = f2_pack(ex2_approx(-r0), ex2_approx(-r1));
    const unsigned long long t = f2_fma(acc[e], c2, f2_fma(f2_pack(r0, r1), c1, c0));
    kv[e] = f2_mul(t, ex);
  }
}


// The exponent e_r of a candidate row's K* scale (kstar_scale_exp of the
// row's bound on K*): the outputscale for the Matern-5/2 kernel; for the
// composite kernel s2 + s2_x + s2_c w* max_j w_j (each factor k52, k32 <= 1).
// Builders, the epilogue and the K* kernel all derive it here.
__device__ __forceinline__ int row_exp(int kern, const float *par, float ws) {
  float bound = par[kParS2];
  if (kern) bound = fmaf(par[kParS2c] * ws, par[kParWmax], par[kParS2] + par[kParS2x]);
  if (!(bound > 0.f) || !(bound < 3.0e38f)) bound = 1.f;
  return kstar_scale_exp(bound);
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

// The mean of a candidate is recomputed in fp64 when its terms K*_j alpha_j
// add up to more than kFixRatio times the mean's scale max(|mean|, s): the
// fp32 cross-covariance's rounding (a few units in the last place per entry,
// amplified by that ratio) would otherwise exceed the 1e-5 tolerance. Below
// the ratio the fp32 mean's error stays under about 6e-6 of the scale.
constexpr float kFixRatio = 256.f;

// A row's mean in fp64 for the Matern-5/2 kernel, computed by a whole warp
// (lane = column j mod 32) and returned to every lane: the candidate's
// coordinates scaled by 1/l as hi + lo, the training points' x / l as hi + lo
// and alpha as hi + lo, read from the side input in global memory (the rare,
// exact path; the warp takes one flagged row at a time).
template <int DP>
__device__ double mean_fp64_warp(const float *xrow, int d, const float *x0, int cf, int n,
                                 int lane) {
  const float *il = x0 + xt_param_offset(DP);
  const double s2 = il[2 * DP + kParS2];
  // lane k holds the candidate's coordinate k scaled by 1/l
  const double xs_l = lane < d ? (double)xrow[lane] * ((double)il[lane] + (double)il[DP + lane]) : 0.0;
  double acc = 0.0;
  for (int j0 = 0; j0 < n; j0 += 32) {
    const int j = j0 + lane;
    const float *ch = x0 + (size_t)(min(j, n - 1) / BOUTE_KCHUNK) * cf;
    const int jj = j % BOUTE_KCHUNK;
    double r2 = 0.0;
    for (int k = 0; k < d; ++k) {
      const double xs = __shfl_sync(0xffffffffu, xs_l, k);
      const double df =
          xs - ((double)ch[k * BOUTE_KCHUNK + jj] + (double)ch[(DP + k) * BOUTE_KCHUNK + jj]);
      r2 = fma(df, df, r2);
    }
    if (j >= n) continue;
    const double r = sqrt(r2) / kCoordScale52;  // (the side input's scale)
    const double kv = s2 * (1.0 + 2.2360679774997896964 * r + (5.0 / 3.0) * (r * r)) *
                      exp(-2.2360679774997896964 * r);
    const float *al = ch + xt_alpha_offset(DP) + jj;  // alpha hi, lo
    acc = fma(kv, (double)al[0] + (double)al[BOUTE_KCHUNK], acc);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  return acc;
}

// The work sequence every role follows: per unit (tile, objective), the
// groups of up to kGroup blocks; per group the chunks [0, kc[last block]).
struct Groups {
  int n;  // groups per unit
  __device__ __forceinline__ explicit Groups(const PostPlan &p) : n((p.nblk + kGroup - 1) / kGroup) {}
  __device__ __forceinline__ static int first(int g) { return g * kGroup; }
  __device__ __forceinline__ static int last(const PostPlan &p, int g) {
    return min(p.nblk, (g + 1) * kGroup) - 1;
  }
  // chunks [0, prev(g)) were built by an earlier group
  __device__ __forceinline__ static int prev(const PostPlan &p, int g) {
    return g > 0 ? p.kc[last(p, g - 1)] : 0;
  }
  // The chunk at position i of a group's sequence of kcg chunks. With cached
  // chunks (mix) the new chunks [kcp, kcg) alternate with the cached ones
  // [0, kcp), so that the builders always have a chunk to build while the
  // tensor cores work through the cached ones; otherwise in order.
  __device__ __forceinline__ static int chunk_at(int i, int kcp, int kcg, bool mix) {
    if (!mix) return i;
    const int nb = kcg - kcp, m = min(nb, kcp);
    if (i < 2 * m) return (i & 1) ? (i >> 1) : kcp + (i >> 1);
    return nb > kcp ? kcp + (i - m) : i - m;
  }
};

// PRE: the K* values come precomputed (kstar_kernel, scaled fp32 images)
// instead of being built here; everything else is the same. KERN: the
// handle's kernel (0 Matern-5/2, 1 composite), which the builders evaluate
// (!PRE) and from which every role derives the rows' K* scale.
template <int DP, bool PRE, int KERN = 0>
__global__ void __launch_bounds__(Layout<DP>::kThreads, 1)
    posterior_kernel(const __grid_constant__ PostArgs a) {
  constexpr int kBldWarps = Layout<DP>::kBld;
  constexpr int COLS = Layout<DP>::kCols;   // columns of a half per builder thread
  // 8 builder warps building the Matern kernel here: each builder thread
  // covers two candidate rows (kstar_pair), so that every training coordinate
  // it loads serves two K* entries (half the shared-memory loads per entry)
  constexpr bool kPair = !PRE && KERN == 0 && kBldWarps == 8;
  constexpr int RP = kPair ? 2 : 1;  // candidate rows per builder thread
  constexpr int CT = COLS / RP;      // its columns of a 32-point half
  constexpr int GPT = 32 / CT;       // column groups (partial means per row)
  constexpr int RPT = 32 / GPT;      // builder threads of a warp along the rows
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment (the 128-byte swizzle atom) as an offset from the
  // shared array, so that every access below stays a shared-memory access
  uint8_t *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const PostPlan &pl = a.plan;
  const int n = a.n, m = a.m, d = a.d, SA = a.sa, SB = a.sb, SX = a.sx;
  const int cf = xt_chunk_floats(DP);
  const Groups grp(pl);

  uint8_t *ring_b = sm + (size_t)SA * kABytes;
  uint8_t *ring_x = ring_b + (size_t)SB * a.b_bytes;
  uint8_t *ring_s = ring_x + (size_t)SX * a.x_bytes;  // PRE staging (SA stages)
  uint64_t *bars = (uint64_t *)(ring_s + (PRE ? (size_t)SA * kStageBytes : 0));
  uint64_t *a_full = bars, *a_empty = bars + kMaxA;
  uint64_t *b_full = bars + 2 * kMaxA, *b_empty = b_full + kMaxB;
  uint64_t *x_full = b_full + 2 * kMaxB, *x_empty = x_full + kMaxX;
  uint64_t *acc_full = x_full + 2 * kMaxX, *acc_empty = acc_full + kSlots;
  uint64_t *drain = acc_empty + kSlots;
  uint64_t *st_full = drain + 1, *st_empty = st_full + kMaxA;  // PRE staging
  uint64_t *cache_ready = st_empty + kMaxA;  // a group's K* chunks are stored
  // the builders' partial means of a unit are written / read by the epilogue
  uint64_t *mean_ready = cache_ready + 1, *mean_empty = mean_ready + 1;
  uint32_t *tmem_holder = (uint32_t *)(mean_empty + 1);
  volatile int *abort = (volatile int *)(tmem_holder + 1);
  // after the 512-byte barrier area: per column group and row of the tile,
  // a builder thread's partial mean (hi, lo) and magnitude sum
  float *red = (float *)(bars + 64);

  auto a_hi = [&](int s) { return sm + (size_t)s * kABytes; };
  auto b_reg = [&](int s) { return ring_b + (size_t)s * a.b_bytes; };
  auto xt_reg = [&](int j) { return (float *)(ring_x + (size_t)j * a.x_bytes); };
  auto stage = [&](int s) { return (const float *)(ring_s + (size_t)s * kStageBytes); };

  if (tid == 0) {
    for (int s = 0; s < kMaxA; ++s) {
      mbar_init(&a_full[s], kBldWarps);
      mbar_init(&a_empty[s], 1);
      mbar_init(&st_full[s], 1);
      mbar_init(&st_empty[s], kBldWarps);
    }
    for (int s = 0; s < kMaxB; ++s) {
      mbar_init(&b_full[s], 1);
      mbar_init(&b_empty[s], 1);
    }
    for (int j = 0; j < kMaxX; ++j) {
      mbar_init(&x_full[j], 1);
      mbar_init(&x_empty[j], kBldWarps);
    }
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(cache_ready, 1);
    mbar_init(mean_ready, kBldWarps);
    mbar_init(mean_empty, kEpiWarps);
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
  const int units = a.tiles_total * m;

  constexpr bool kSep = Layout<DP>::kSepCache;
  constexpr int kBldWarp0 = Layout<DP>::kBldWarp0;
  if (warp == 0 || warp == kXtWarp || (kSep && warp == kCacheWarp)) {
    // ------------------------------------ producers (B / side input / cached K* chunks)
    // With a warp of their own for the cached chunks, waiting for the A stage
    // of a cached chunk never holds up the side input of the new ones.
    if (lane == 0 && (warp != kCacheWarp || a.ncache > 0)) {
      const bool is_b = warp == 0;
      const int R = is_b ? SB : SX;
      uint64_t *full = is_b ? b_full : x_full, *empty = is_b ? b_empty : x_empty;
      const bool with_st = PRE && warp == kXtWarp;  // the side-input producer also stages K*
      const bool with_cache = a.ncache > 0 && warp == (kSep ? kCacheWarp : kXtWarp);
      uint32_t q = 0, qa = 0, nready = 0;
      RingPos rp, ra;
      int last_q = -1, last_qa = -1;  // last jobs issued
      int last_ca = -1;               // last cached-chunk copy (A ring position)
      for (int unit = blockIdx.x; unit < units && !*abort; unit += gridDim.x) {
        const int tile = unit / m, t = unit % m;
        const int bt = (tile / a.tiles_per_problem) * m + t;
        for (int g = 0; g < grp.n && !*abort; ++g) {
          const int q0 = Groups::first(g), q1 = Groups::last(pl, g), kcg = pl.kc[q1];
          const int kcp = Groups::prev(pl, g);
          if (with_cache && kcp > 0) {  // the earlier groups' stores have landed
            if (!wait_or_abort(cache_ready, nready & 1u, abort)) break;
            ++nready;
            fence_proxy_async_global();
          }
          const bool mix = a.ncache > 0 && kcp > 0;
          for (int i = 0; i < kcg && !*abort; ++i) {
            const int c = Groups::chunk_at(i, kcp, kcg, mix);
            if (with_cache) {  // the A ring's positions; the cached chunks' A stages
              const int s = ra.idx;
              const bool cached = c < kcp;
              if (cached) {  // the A stage from this CTA's cache
                if (qa >= (uint32_t)SA && !wait_or_abort(&a_empty[s], ra.phase ^ 1u, abort)) break;
                mbar_expect_tx(&a_full[s], kABytes);
                if (BOUTE_INB(blockIdx.x * a.ncache + c, (long long)gridDim.x * a.ncache))
                  bulk_g2s(a_hi(s),
                           a.kcache + ((size_t)blockIdx.x * a.ncache + c) * (kABytes / 2),
                           kABytes, &a_full[s]);
                mbar_arrive_n(&a_full[s], kBldWarps);
                last_ca = (int)qa;
              }
              ++qa;
              ra.advance(SA);
              if (cached || kSep) continue;  // (the cache warp does nothing else)
            }
            if (!is_b && mix && c < kcp) continue;  // a cached chunk needs no side input
            if (with_st) {  // the chunk's fp32 K* image
              const int s = ra.idx;
              if (qa >= (uint32_t)SA && !wait_or_abort(&st_empty[s], ra.phase ^ 1u, abort)) break;
              mbar_arrive_expect_tx(&st_full[s], kStageBytes);
              if (BOUTE_INB((long long)unit * pl.nchunk + c, (long long)units * pl.nchunk))
                bulk_g2s((void *)stage(s),
                         a.kst + ((size_t)unit * pl.nchunk + c) * (kStageBytes / 4), kStageBytes,
                         &st_full[s]);
              last_qa = (int)qa;
              ++qa;
              ra.advance(SA);
            }
            // B: one stage per block of the group that needs chunk c; side
            // input: the chunk's two 32-point halves
            const int jobs = is_b ? q1 - q0 + 1 : 2;
            for (int job = 0; job < jobs; ++job) {
              const int qb = q0 + job;
              if (is_b && pl.kc[qb] <= c) continue;
              const int s = rp.idx;
              if (q >= (uint32_t)R && !wait_or_abort(&empty[s], rp.phase ^ 1u, abort)) break;
              if (is_b) {
                const int ncol = pl.ncol[qb];
                const uint32_t bytes = (uint32_t)(2 * ncol * 128);
                mbar_arrive_expect_tx(&full[s], bytes);
                const long long bo = (long long)bt * pl.image_halves + pl.off[qb] +
                                     (long long)c * 2 * ncol * BOUTE_ACHUNK;
                if (BOUTE_INB(bo + bytes / 2 - 1, (long long)a.B * m * pl.image_halves) &&
                    BOUTE_INB(bytes, (long long)a.b_bytes + 1))
                  bulk_g2s(b_reg(s), a.bop + bo, bytes, &full[s]);
              } else {
                mbar_arrive_expect_tx(&full[s], a.x_bytes);
                const long long xo = ((long long)bt * pl.nxt + 2 * c + job) * cf;
                if (BOUTE_INB(xo + a.x_bytes / 4 - 1, (long long)a.B * m * pl.nxt * cf))
                  bulk_g2s(xt_reg(s), a.xt + xo, a.x_bytes, &full[s]);
              }
              last_q = (int)q;
              ++q;
              rp.advance(R);
            }
          }
        }
      }
      if (*abort) {  // let our copies land before the block exits
        for (int j = std::max(0, last_q - R + 1); j <= last_q; ++j)
          mbar_wait(&full[j % R], (j / R) & 1);
        for (int j = std::max(0, last_qa - SA + 1); j <= last_qa; ++j)
          mbar_wait(&st_full[j % SA], (j / SA) & 1);
        if (last_ca >= 0) mbar_wait(&a_full[last_ca % SA], (last_ca / SA) & 1);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      // the block at position P of this CTA's sequence uses slot P % 4 for
      // the (P / 4)-th time: it waits for that slot's previous use to drain
      uint32_t blkseq = 0;
      bool issued = false;
      RingPos pa, pb;
      for (int unit = blockIdx.x; unit < units && !*abort; unit += gridDim.x) {
        for (int g = 0; g < grp.n && !*abort; ++g) {
          const int q0 = Groups::first(g), q1 = Groups::last(pl, g), kcg = pl.kc[q1];
          const int kcp = Groups::prev(pl, g);
          const bool storing = a.ncache > 0 && g < grp.n - 1;  // a later group needs them
          const bool mix = a.ncache > 0 && kcp > 0;
          uint32_t done = 0;  // chunks issued per block of the group, 5 bits each
          for (int i = 0; i < kcg && !*abort; ++i) {
            const int c = Groups::chunk_at(i, kcp, kcg, mix);
            const int sa = pa.idx;
            if (!wait_or_abort(&a_full[sa], pa.phase, abort)) break;
            const uint32_t sah = smem_u32(a_hi(sa)), sal = sah + kAPartBytes;
            const bool store = storing && c >= kcp;  // built here, needed later
            if (store) {
              if (BOUTE_INB(blockIdx.x * a.ncache + c, (long long)gridDim.x * a.ncache))
                bulk_s2g(a.kcache + ((size_t)blockIdx.x * a.ncache + c) * (kABytes / 2),
                         a_hi(sa), kABytes);
              bulk_commit();
            }
            for (int jb = 0; jb <= q1 - q0; ++jb) {
              const int qb = q0 + jb;
              if (pl.kc[qb] <= c) continue;
              const uint32_t P = blkseq + (uint32_t)jb;
              const int sl = (int)(P % kSlots);
              const int nd = (int)((done >> (5 * jb)) & 31u);  // chunks of this block issued
              done += 1u << (5 * jb);
              if (nd == 0 && P >= kSlots &&
                  !wait_or_abort(&acc_empty[sl], (P / kSlots - 1) & 1, abort))
                break;
              const int sb = pb.idx;
              if (!wait_or_abort(&b_full[sb], pb.phase, abort)) break;
              tc_fence_after();
              const int ncol = pl.ncol[qb];
              const uint32_t idesc = idesc_f16(ncol);
              const uint32_t dtm = tmem + (uint32_t)(sl * BOUTE_BLKCOLS);
              const uint32_t sbh = smem_u32(b_reg(sb)), sbl = sbh + ncol * 128;
#pragma unroll
              for (int ks = 0; ks < 4; ++ks) {
                const uint64_t dah = sdesc_sw128(sah + ks * 32), dal = sdesc_sw128(sal + ks * 32);
                const uint64_t dbh = sdesc_sw128(sbh + ks * 32), dbl = sdesc_sw128(sbl + ks * 32);
                mma_f16(dtm, dah, dbh, idesc, (nd > 0 || ks > 0) ? 1u : 0u);
                mma_f16(dtm, dah, dbl, idesc, 1u);
                mma_f16(dtm, dal, dbh, idesc, 1u);
              }
              mma_commit(&b_empty[sb]);
              pb.advance(SB);
              if (nd == pl.kc[qb] - 1) mma_commit(&acc_full[sl]);  // the block is complete
              issued = true;
            }
            if (*abort) break;
            if (store) bulk_wait_read();  // the stage is read before it is reused
            mma_commit(&a_empty[sa]);
            pa.advance(SA);
          }
          if (storing && !*abort) {  // the group's chunks are in the cache
            bulk_wait();
            mbar_arrive_count(cache_ready);
          }
          blkseq += (uint32_t)(q1 - q0 + 1);
        }
      }
      if (issued) {  // every MMA of ours has completed before TMEM is released
        mma_commit(drain);
        mbar_wait(drain, 0);
      }
      bulk_wait();  // and every store of ours
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ---------------------------------------------------------------- epilogue
    const int eq = warp & 3;  // TMEM lane quarter this warp may access
    uint32_t blkseq = 0, nmean = 0;
    const uint32_t lanes = (uint32_t)(32 * eq) << 16;
    for (int unit = blockIdx.x; unit < units && !*abort; unit += gridDim.x) {
      const int tile = unit / m, t = unit % m;
      const int b = tile / a.tiles_per_problem;
      const long long row =
          (long long)(tile % a.tiles_per_problem) * BOUTE_TILE_M + 32 * eq + lane;
      const bool live = row < a.N;
      const float *par = a.xt + (size_t)(b * m + t) * pl.nxt * cf + xt_param_offset(DP) + 2 * DP;
      float prior = a.s2f[b * m + t], ws = 0.f;
      if (a.kern && live) {  // composite kernel: k(x, x) = s2 + s2_x + s2_c w(x)^2
        const float *c0 = a.xt + (size_t)(b * m + t) * pl.nxt * cf;
        const float *bp = chunk_pref(c0, DP), *xrow = a.Xc + ((size_t)b * a.N + row) * d;
        float e = 0.f;
        for (int k = 0; k < d; ++k) e = fmaf(bp[k], xrow[k], e);
        ws = expf(e);
        prior = fmaf(par[kParS2c] * ws, ws, prior);
      }
      // the row's K* scale 2^e_r; the in-sample shifts (G blocks) leave with
      // 2^-(e_r + e_G) applied
      const int er = row_exp(a.kern, par, ws);
      const float gscale = pl.S_in > 0 ? exp2i(-(er + (int)par[kParEG])) : 0.f;
      float* shrow = pl.S_in > 0 ? a.shift + (size_t)(b * m + t) * pl.S_in * a.N + row : nullptr;
      float ss = 0.f, ssh = 0.f;  // W's and H^T's sums of squares
      for (int g = 0; g < grp.n && !*abort; ++g) {
        const int q0 = Groups::first(g), q1 = Groups::last(pl, g);
        for (int qb = q0; qb <= q1; ++qb) {
          const uint32_t P = blkseq + (uint32_t)(qb - q0);
          const int sl = (int)(P % kSlots);
          if (!wait_or_abort(&acc_full[sl], (P / kSlots) & 1, abort)) break;
          tc_fence_after();
          const uint32_t ta = tmem + (uint32_t)(sl * BOUTE_BLKCOLS) + lanes;
          if (qb < pl.nwblk + pl.nhblk) {
            float sq = 0.f;
            for (int cc = 0; cc < pl.ncol[qb]; cc += 16) {
              float v[16];
              tmem_ld16(ta + cc, v);
#pragma unroll
              for (int e = 0; e < 16; ++e) sq = fmaf(v[e], v[e], sq);  // zero beyond n
            }
            if (qb < pl.nwblk) ss += sq;
            else ssh += sq;
          } else {  // G block: the shifts of draws s0 .. s0 + ncol
            const int s0 = BOUTE_BLKCOLS * (qb - pl.nwblk - pl.nhblk);
            for (int cc = 0; cc < pl.ncol[qb]; cc += 16) {
              float v[16];
              tmem_ld16(ta + cc, v);
              if (live)
#pragma unroll
                for (int e = 0; e < 16; ++e)
                  if (s0 + cc + e < pl.S_in &&
                      BOUTE_INB((((long long)b * m + t) * pl.S_in + s0 + cc + e) * a.N + row,
                                (long long)a.B * m * pl.S_in * a.N))
                    shrow[(size_t)(s0 + cc + e) * a.N] = v[e] * gscale;
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_count(&acc_empty[sl]);
        }
        blkseq += (uint32_t)(q1 - q0 + 1);
      }
      if (*abort) break;
      // the mean: the builders' partials of this row, one per column group,
      // added in order with error-free sums; its terms reach hundreds of times
      // the result when K is ill-conditioned, and their magnitudes
      // sum_j K*_j |alpha_j| decide whether the row is recomputed in fp64
      if (!wait_or_abort(mean_ready, nmean & 1u, abort)) break;
      ++nmean;
      float mhi = 0.f, mlo = 0.f, mag = 0.f;
#pragma unroll
      for (int q = 0; q < GPT; ++q) {
        const float *rp = red + ((size_t)q * BOUTE_TILE_M + 32 * eq + lane) * 3;
        float e;
        two_sum_f(mhi, rp[0], mhi, e);
        mlo += rp[1] + e;
        mag += rp[2];
      }
      __syncwarp();
      if (lane == 0) mbar_arrive_count(mean_empty);
      float mean = ldexpf(mhi + mlo, -er);
      if (KERN == 0) {  // ill-conditioned rows: the mean in fp64, one row at a time
        const float sc = ldexpf(sqrtf(par[kParS2]), er);  // the mean's scale, scaled like K*
        const bool fix = live && mag > kFixRatio * fmaxf(fabsf(mhi), sc);
        unsigned todo = __ballot_sync(0xffffffffu, fix);
        while (todo) {
          const int src = __ffs(todo) - 1;
          todo &= todo - 1;
          const long long rr = (long long)(tile % a.tiles_per_problem) * BOUTE_TILE_M + 32 * eq + src;
          const float *x0 = a.xt + (size_t)(b * m + t) * pl.nxt * cf;
          const double v = mean_fp64_warp<DP>(a.Xc + ((long long)b * a.N + rr) * d, d, x0, cf, n,
                                              lane);
          if (lane == src) mean = (float)v;
        }
      }
      if (live && BOUTE_INB(((long long)b * m + t) * a.N + row, (long long)a.B * m * a.N))
        a.mean[((size_t)b * m + t) * a.N + row] = mean;
      if (live) {
        // V carries the scales 2^e_r (K*) and 2^e_W (W); H^T k* 2^e_r and 2^e_H
        float vv = prior - ldexpf(ss, -2 * (er + (int)par[kParEW]));
        if (pl.nhblk > 0) vv -= ldexpf(ssh, -2 * (er + (int)par[kParEH]));
        if (BOUTE_INB(((long long)b * m + t) * a.N + row, (long long)a.B * m * a.N))
          a.var[((size_t)b * m + t) * a.N + row] = vv > 0.f ? vv : 0.f;
      }
    }
  } else if (warp >= kBldWarp0) {
    // ---------------------------------------------------------------- K* builders
    // thread -> (row r, and r + RPT with rows in pairs; column group g): CT
    // consecutive columns of each half, RPT threads x GPT column groups per
    // warp (a layout with 32 rows of one column group per warp, whose
    // coordinate loads are broadcasts, measured slower: those loads cost more
    // shared-memory wavefronts, not fewer)
    const int bw = warp - kBldWarp0;
    const int r = bw * (RPT * RP) + lane % RPT, g = lane / RPT;  // rows r (and r + RPT)
    uint32_t nmean = 0;
    RingPos pa, px;
    uint32_t qa = 0;
    for (int unit = blockIdx.x; unit < units && !*abort; unit += gridDim.x) {
      const int tile = unit / m;
      const int b = tile / a.tiles_per_problem;
      const long long row = (long long)(tile % a.tiles_per_problem) * BOUTE_TILE_M + r;
      float xr[DP];  // (unused with rows in pairs)
      unsigned long long xs2[DP];
      float s2 = 0.f;
      CompIn ci{};
      int er = 0;
      if constexpr (kPair) {
        // both rows' scaled coordinates now, with the objective's scales read
        // from the side input in global memory, so that the raw coordinates
        // die here instead of living through the chunk loop
        const float *il = a.xt + (size_t)(b * m + unit % m) * pl.nxt * cf + xt_param_offset(DP);
        er = row_exp(0, il + 2 * DP, 0.f);
        s2 = ldexpf(il[2 * DP + kParS2], er);
        float x0[DP], x1[DP];
        const long long row1 = row + RPT;
        const float *xrow = a.Xc + ((long long)b * a.N + row) * d;
        const float *xrow1 = a.Xc + ((long long)b * a.N + row1) * d;
#pragma unroll
        for (int k = 0; k < DP; ++k) {
          x0[k] = (k < d && row < a.N) ? xrow[k] : 0.f;
          x1[k] = (k < d && row1 < a.N) ? xrow1[k] : 0.f;
        }
        scaled_pair<DP>(x0, x1, il, xs2);
      } else if (!PRE || KERN == 1) {
        const float *xrow = a.Xc + ((long long)b * a.N + row) * d;
#pragma unroll
        for (int k = 0; k < DP; ++k) xr[k] = (k < d && row < a.N) ? xrow[k] : 0.f;
      }
      // the mean K* alpha: its terms reach hundreds of times the result when K
      // is ill-conditioned, so they are summed with compensation, and their
      // magnitudes sum_j K*_j |alpha_j| decide whether the row needs the fp64 path
      Kahan2 mu2;
      unsigned long long mag2 = 0ull;
      for (int gi = 0; gi < grp.n && !*abort; ++gi) {
        const int kcg = pl.kc[Groups::last(pl, gi)], kcp = Groups::prev(pl, gi);
        // with the cache every built chunk is new and adds to the mean;
        // without it the last group builds every chunk and adds them all
        const bool mix = a.ncache > 0 && kcp > 0;
        const bool mean_grp = a.ncache > 0 || gi == grp.n - 1;
        for (int i = 0; i < kcg && !*abort; ++i, ++qa, pa.advance(SA)) {
          const int c = mix ? Groups::chunk_at(i, kcp, kcg, true) : i;
          if (mix && c < kcp) continue;  // cached: the producer brings it
          const int s = pa.idx;
          if (qa >= (uint32_t)SA && !wait_or_abort(&a_empty[s], pa.phase ^ 1u, abort)) break;
          if (PRE && !wait_or_abort(&st_full[s], pa.phase, abort)) break;
          uint8_t *Ah = a_hi(s), *Al = Ah + kAPartBytes;
          for (int h = 0; h < 2; ++h, px.advance(SX)) {
            const int j = px.idx;
            if (!wait_or_abort(&x_full[j], px.phase, abort)) break;
            const float *xth = xt_reg(j);
            const float *alp = xth + xt_alpha_offset(DP);
            if (!kPair && gi == 0 && c == 0 && h == 0) {  // new objective: its parameters came with the chunk
              const float *il = xth + xt_param_offset(DP);
              const float *par = il + 2 * DP;
              if (KERN == 1) ci = chunk_comp(xth, DP);
              const float ws = KERN == 1 ? cand_weight<DP>(xr, chunk_pref(xth, DP)) : 0.f;
              er = row_exp(KERN, par, ws);
              if (!PRE) {
                scaled_candidate<DP>(xr, il, xs2);
                s2 = ldexpf(par[kParS2], er);
                if (KERN == 1) {
                  ci.ws = ws;
                  ci.s2c = ldexpf(ci.s2c, er);
                  ci.s2x = ldexpf(ci.s2x, er);
                }
              }
            }
            if constexpr (kPair) {
              const int col0 = BOUTE_KCHUNK * h + CT * g;  // first column within the chunk
              unsigned long long kvp[CT];  // (row r, row r + RPT) per column
              kstar_pair<DP, CT>(xs2, xth, g, s2, kvp);
              const int jbase = BOUTE_ACHUNK * c + col0;
              const float *alg = alp + CT * g;
              // both rows' CT = 8 columns into the A stage as fp16 hi/lo, the
              // mean's terms summed per row; a ragged last half zeroes the
              // columns beyond n
              auto emit2 = [&](auto ragged) {
                static_assert(CT == 8, "one 16-byte store per row and part");
                uint32_t hi[2][4], lo[2][4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const int kk = 2 * e;
                  unsigned long long va = kvp[kk], vb = kvp[kk + 1];
                  if (decltype(ragged)::value) {
                    va = (jbase + kk < n) ? va : 0ull;
                    vb = (jbase + kk + 1 < n) ? vb : 0ull;
                  }
                  if (mean_grp) {  // (each chunk's terms once)
                    const float a0 = alg[kk], a1 = alg[kk + 1];
                    mu2.add(f2_mul(va, f2_dup(a0)));
                    mu2.add(f2_mul(vb, f2_dup(a1)));
                    mag2 = f2_fma(va, f2_dup(fabsf(a0)), mag2);  // (K* >= 0)
                    mag2 = f2_fma(vb, f2_dup(fabsf(a1)), mag2);
                  }
                  float a_0, a_1, b_0, b_1;
                  f2_split(va, a_0, a_1);
                  f2_split(vb, b_0, b_1);
                  split_f16x2(a_0, b_0, hi[0][e], lo[0][e]);
                  split_f16x2(a_1, b_1, hi[1][e], lo[1][e]);
                }
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                  const int o = sw128_off16(r + q * RPT, col0) * 2;  // bytes
                  if (BOUTE_INB(o + 15, (long long)kAPartBytes)) {
                    *(uint4 *)(Ah + o) = make_uint4(hi[q][0], hi[q][1], hi[q][2], hi[q][3]);
                    *(uint4 *)(Al + o) = make_uint4(lo[q][0], lo[q][1], lo[q][2], lo[q][3]);
                  }
                }
              };
              if (jbase + CT <= n) emit2(std::false_type{});
              else emit2(std::true_type{});
            } else {
              float kv[COLS];
              const int col0 = BOUTE_KCHUNK * h + COLS * g;  // first column within the chunk
              if (PRE) {  // this thread's COLS values, from the staged fp32 image
#pragma unroll
                for (int e = 0; e < COLS / 4; ++e) {
                  const float4 v = *(const float4 *)(stage(s) + st_off32(r, col0 + 4 * e));
                  kv[4 * e] = v.x;
                  kv[4 * e + 1] = v.y;
                  kv[4 * e + 2] = v.z;
                  kv[4 * e + 3] = v.w;
                }
              } else {
                kstar_cols<DP, COLS, KERN>(xs2, xth, g, s2, kv, ci);
              }
              const int jbase = BOUTE_ACHUNK * c + col0;
              const float *alg = alp + COLS * g;
              // kernel values of this thread's COLS columns into the A stage as
              // fp16 hi/lo; a ragged last half zeroes the columns beyond n
              auto emit = [&](auto ragged) {
#pragma unroll
                for (int u = 0; u < COLS / 8; ++u) {
                  uint32_t hi[4], lo[4];
#pragma unroll
                  for (int e = 0; e < 4; ++e) {
                    const int kk = 8 * u + 2 * e;
                    float v0 = kv[kk], v1 = kv[kk + 1];
                    if (decltype(ragged)::value) {
                      v0 = (jbase + kk < n) ? v0 : 0.f;
                      v1 = (jbase + kk + 1 < n) ? v1 : 0.f;
                    }
                    if (mean_grp) {  // (each chunk's terms once)
                      const unsigned long long v2 = f2_pack(v0, v1);
                      const unsigned long long a2 = *(const unsigned long long *)(alg + kk);
                      mu2.add(f2_mul(v2, a2));
                      mag2 = f2_fma(v2, a2 & 0x7fffffff7fffffffull, mag2);  // (K* >= 0)
                    }
                    split_f16x2(v0, v1, hi[e], lo[e]);
                  }
                  const int o = sw128_off16(r, col0 + 8 * u) * 2;  // bytes
                  if (BOUTE_INB(o + 15, (long long)kAPartBytes)) {
                    *(uint4 *)(Ah + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                    *(uint4 *)(Al + o) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
                  }
                }
              };
              if (jbase + COLS <= n) emit(std::false_type{});
              else emit(std::true_type{});
            }
            __syncwarp();
            if (lane == 0) mbar_arrive_count(&x_empty[j]);
          }
          if (*abort) break;
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive_count(&a_full[s]);
            if (PRE) mbar_arrive_count(&st_empty[s]);
          }
        }
      }
      if (*abort) break;
      // the thread's sum as a float pair (hi, lo) and its magnitude sum, for
      // the epilogue (the buffer is free once it has read the previous unit's)
      float se, so, ce, co, me, mo;
      f2_split(mu2.s, se, so);
      f2_split(mu2.c, ce, co);
      f2_split(mag2, me, mo);
      if (nmean > 0 && !wait_or_abort(mean_empty, (nmean - 1) & 1u, abort)) break;
      ++nmean;
      float *rp = red + ((size_t)g * BOUTE_TILE_M + r) * 3;
      if constexpr (kPair) {  // the pair's lanes are the two rows, each a Kahan sum s - c
        float *rq = red + ((size_t)g * BOUTE_TILE_M + r + RPT) * 3;
        rp[0] = se;
        rp[1] = -ce;
        rp[2] = me;
        rq[0] = so;
        rq[1] = -co;
        rq[2] = mo;
      } else {  // the pair's lanes are two sets of the row's columns
        float hi, lo;
        two_sum_f(se, so, hi, lo);
        lo -= ce + co;
        rp[0] = hi;
        rp[1] = lo;
        rp[2] = me + mo;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive_count(mean_ready);
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
              float *var, cudaStream_t s, float *shift) {
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
  a.shift = shift;
  if (!shift && a.plan.S_in > 0) {  // the plain posterior: W's blocks only
    a.plan.nblk = a.plan.nwblk;
    a.plan.nhblk = 0;
    a.plan.S_in = 0;
  }
  a.kern = gp->kern;
  // the chunk cache (not with K* precomputed, where no chunk is built)
  a.kcache = gp->kcache;
  const int want = kstar_cache_chunks(a.plan);
  a.ncache =
      (!kst && gp->kcache && gp->kcache_sms >= num_sms() && want <= gp->kcache_cap) ? want : 0;
  a.tiles_per_problem = (int)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M);
  a.tiles_total = a.tiles_per_problem * gp->B;
  int wmax = 0;  // the widest block sizes a B stage
  for (int q = 0; q < a.plan.nblk; ++q) wmax = std::max(wmax, a.plan.ncol[q]);
  a.b_bytes = (uint32_t)(2 * wmax * 128);
  a.x_bytes = (uint32_t)round_up(xt_chunk_floats(DP) * 4, 16);
  // alignment slack, barriers, TMEM address, flag; the partial means (twice
  // the column groups where the builders take rows in pairs)
  const bool pair = !kst && !gp->kern && Layout<DP>::kBld == 8;
  const size_t fixed =
      1024 + 512 + (size_t)(32 / Layout<DP>::kCols) * (pair ? 2 : 1) * BOUTE_TILE_M * 3 * 4;
  const size_t budget = 227 * 1024 - fixed;
  const size_t st = kst ? kStageBytes : 0;  // staging beside each A stage (PRE)
  // K* stages before B stages: a deeper A ring lets the builders run ahead of
  // the tensor cores through the groups where the MMAs outweigh the building
  // (measured best: 4 A + 2 B stages with 8 builder warps, 3 + 3 with 16),
  // then the side input's ring as deep as what is left allows
  a.sx = kMaxX;
  a.sa = Layout<DP>::kBld == 8 ? 4 : 3;
  a.sb = Layout<DP>::kBld == 8 ? 2 : 3;
  while ((size_t)a.sa * (kABytes + st) + (size_t)a.sb * a.b_bytes + (size_t)a.sx * a.x_bytes >
         budget) {
    if (a.sx > 4) --a.sx;
    else if (a.sa > 2) --a.sa;
    else if (a.sb > 2) --a.sb;
    else if (a.sx > 2) --a.sx;
    else return BOUTE_ERR_UNSUPPORTED;
  }
  const size_t smem = fixed + (size_t)a.sa * (kABytes + st) + (size_t)a.sb * a.b_bytes +
                      (size_t)a.sx * a.x_bytes;
  const int grid = std::max(1, std::min(a.tiles_total * a.m, num_sms()));  // (tile, objective) units
  auto go = [&](auto kern) {
    prefer_shared(kern);
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    launch_pdl(kern, dim3(grid), dim3(Layout<DP>::kThreads), smem, s, a);
  };
  if (kst) {
    if (gp->kern) go(posterior_kernel<DP, true, 1>);
    else go(posterior_kernel<DP, true, 0>);
  } else if (gp->kern) {
    go(posterior_kernel<DP, false, 1>);
  } else {
    go(posterior_kernel<DP, false, 0>);
  }
  count_launch();
  return last_launch_status();
}

// ---- K* ahead of the fit's results ------------------------------------------------
// One block per (tile, objective) unit, threads laid out as the posterior's
// builders: all n training points' K* values of the tile's 128 candidates, in
// the builders' arithmetic and scale (2^e_r), zero beyond n. Each 64-point
// chunk is stored as a 32 KB fp32 image ([128 x 64], st_off32), which the
// posterior brings in with one bulk copy and splits into its fp16 operand
// parts. The training points' side input is staged in shared memory. It needs
// the set-up's side input (not the fit's results) and the candidates.
template <int DP, int KERN>
__global__ void __launch_bounds__(Layout<DP>::kBld * 32) kstar_kernel(
    const float *Xc, const float *xt, long long N, int d, int m, int n, int tiles_per_problem,
    int nxt, float *kst) {
  constexpr int COLS = Layout<DP>::kCols, GPR = 32 / COLS, RPW = 32 / GPR;
  extern __shared__ __align__(16) float xs[];  // nxt side-input chunks
  __shared__ float wmax_s;
  const int unit = blockIdx.x, tile = unit / m, t = unit % m, b = tile / tiles_per_problem;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = warp * RPW + lane % RPW, g = lane / RPW;
  const long long row = (long long)(tile % tiles_per_problem) * BOUTE_TILE_M + r;
  const int cf = xt_chunk_floats(DP);  // a multiple of 4
  const float4 *x4 = (const float4 *)(xt + (size_t)(b * m + t) * nxt * cf);
  for (int e = threadIdx.x; e < nxt * cf / 4; e += blockDim.x) ((float4 *)xs)[e] = x4[e];
  const float *xrow = Xc + ((long long)b * N + row) * d;
  float xr[DP];
#pragma unroll
  for (int k = 0; k < DP; ++k) xr[k] = (k < d && row < N) ? xrow[k] : 0.f;
  __syncthreads();
  const float *il = xs + xt_param_offset(DP);
  float par[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) par[k] = il[2 * DP + k];
  if (KERN == 1) {  // the largest training-point preference weight (as the fit finds it)
    if (warp == 0) {
      float wm = 0.f;
      for (int j = lane; j < n; j += 32)
        wm = fmaxf(wm, xs[(size_t)(j / BOUTE_KCHUNK) * cf + BOUTE_KCHUNK * DP + j % 32]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
      if (lane == 0) wmax_s = wm;
    }
    __syncthreads();
    par[kParWmax] = wmax_s;
  }
  unsigned long long xs2[DP];
  scaled_candidate<DP>(xr, il, xs2);
  CompIn ci{};
  float ws = 0.f;
  if (KERN == 1) {
    ci = chunk_comp(xs, DP);
    ws = cand_weight<DP>(xr, chunk_pref(xs, DP));
  }
  const int er = row_exp(KERN, par, ws);
  const float s2 = ldexpf(par[kParS2], er);
  if (KERN == 1) {
    ci.ws = ws;
    ci.s2c = ldexpf(ci.s2c, er);
    ci.s2x = ldexpf(ci.s2x, er);
  }
  for (int c = 0; c < nxt; ++c) {  // 32-point halves
    float kv[COLS];
    kstar_cols<DP, COLS, KERN>(xs2, xs + (size_t)c * cf, g, s2, kv, ci);
    const int jbase = c * BOUTE_KCHUNK + COLS * g;
#pragma unroll
    for (int kk = 0; kk < COLS; ++kk) kv[kk] = (jbase + kk < n) ? kv[kk] : 0.f;
    float *img = kst + ((size_t)unit * (nxt / 2) + c / 2) * (kStageBytes / 4);
    const int col0 = BOUTE_KCHUNK * (c & 1) + COLS * g;
#pragma unroll
    for (int g4 = 0; g4 < COLS / 4; ++g4)
      *(float4 *)(img + st_off32(r, col0 + 4 * g4)) =
          make_float4(kv[4 * g4], kv[4 * g4 + 1], kv[4 * g4 + 2], kv[4 * g4 + 3]);
  }
}

template <int DP>
int launch_kstar_dp(const Gp *gp, const float *Xc, long long N, float *kst, cudaStream_t s) {
  const int tpp = (int)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M);
  const int units = tpp * gp->B * gp->m;
  const size_t smem = (size_t)gp->plan.nxt * xt_chunk_floats(DP) * sizeof(float);
  auto go = [&](auto kern) {
    prefer_shared(kern);
    // (set on every launch: the kernel's static array counts against the same
    // 48 KB default as the dynamic part)
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
      return last_launch_status();
    kern<<<units, Layout<DP>::kBld * 32, smem, s>>>(Xc, gp->xt, N, gp->d, gp->m, gp->n, tpp,
                                                    gp->plan.nxt, kst);
    return (int)BOUTE_OK;
  };
  if (int r = gp->kern ? go(kstar_kernel<DP, 1>) : go(kstar_kernel<DP, 0>)) return r;
  count_launch();
  return last_launch_status();
}

}  // namespace

BOUTE_BOUNDS_READER(posterior)

int launch_posterior_joint(const Gp *gp, const float *Xc, long long N, float *mean, float *cvar,
                           float *shift, cudaStream_t s, const float *kst) {
  if (N <= 0) return BOUTE_OK;
  switch (gp->DP) {
    case 8: return launch_dp<8>(gp, Xc, kst, N, mean, cvar, s, shift);
    case 12: return launch_dp<12>(gp, Xc, kst, N, mean, cvar, s, shift);
    case 16: return launch_dp<16>(gp, Xc, kst, N, mean, cvar, s, shift);
    case 24: return launch_dp<24>(gp, Xc, kst, N, mean, cvar, s, shift);
    case 32: return launch_dp<32>(gp, Xc, kst, N, mean, cvar, s, shift);
  }
  return BOUTE_ERR_UNSUPPORTED;
}

int launch_posterior(const Gp *gp, const float *Xc, long long N, float *mean, float *var,
                     cudaStream_t s, const float *kst) {
  return launch_posterior_joint(gp, Xc, N, mean, var, nullptr, s, kst);
}

int kstar_cache_chunks(const PostPlan &plan) {
  const int ngroup = (plan.nblk + kGroup - 1) / kGroup;
  if (ngroup < 2) return 0;
  const int last_of_prev = std::min(plan.nblk, (ngroup - 1) * kGroup) - 1;
  return plan.kc[last_of_prev];  // every chunk the groups before the last build
}

size_t kstar_floats(const Gp *gp, long long N) {
  const size_t tpp = (size_t)((N + BOUTE_TILE_M - 1) / BOUTE_TILE_M);
  return tpp * gp->B * gp->m * gp->plan.nchunk * (kStageBytes / 4);
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
