// Device helpers shared by the CUDA translation units of libboute:
// bounded mbarrier waits, bulk (TMA-engine) copies, tcgen05 tensor-core and
// tensor-memory wrappers, and the operand-image layout that the fit writes and
// the posterior kernel reads. sm_103a only.
#pragma once

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "boute.h"

#define BOUTE_MAX_D 32       // candidate dimension limit (registers per thread)
#define BOUTE_MAX_M 4        // objectives per problem
#define BOUTE_MAX_N 2048     // training points per problem
#define BOUTE_MAX_BLK 16     // 128-column output blocks of the posterior contraction
#define BOUTE_TILE_M 128     // candidates per posterior tile (MMA M)
#define BOUTE_KCHUNK 32      // training points per side-input chunk
#define BOUTE_ACHUNK 64      // reduction columns per operand chunk (128 B of fp16)
#define BOUTE_BLKCOLS 128    // output columns per accumulator block (one TMEM slot)
#define BOUTE_WAIT_NS 2000000000ull  // bound on any single device-side wait

namespace boute {

// ---------------------------------------------------------------- host/device
// Operand plan of the posterior contraction V = K* W^T, W = L^-1, for one
// (problem, objective): output column i of V is row i of W. Output columns
// come in blocks of 128 (one tensor-memory accumulator slot each; the last
// block's width is n rounded up to 16); the reduction over the training
// points comes in chunks of 64 (one 128-byte row of fp16 per operand row).
// Block q needs the chunks [0, kc[q]) only, because row i of W is zero beyond
// column i. Its operand images follow one another: for each chunk, W's rows of
// the block as fp16 hi then fp16 lo parts (ncol[q] rows x 64 halves each) in
// the swizzled K-major layout tcgen05.mma reads. npad (n rounded up to 32) is
// the fit's padded size; nxt side-input chunks of 32 points (n rounded up to
// 64) cover the nchunk operand chunks. (The mean K* alpha is reduced on the
// CUDA cores while K* is built, in compensated fp32.)
struct PostPlan {
  int n, npad, nxt, nchunk, nblk;
  // blocks [0, nwblk) hold W = L^-1 (lower triangular); with in-sample draws
  // (S_in > 0) the dense blocks of H^T (nhblk, summed squares) and of G^T
  // (the rest, one output column per in-sample draw) follow
  int nwblk, nhblk, S_in;
  int ncol[BOUTE_MAX_BLK], kc[BOUTE_MAX_BLK];
  long long off[BOUTE_MAX_BLK];  // half offset of block q's first chunk image
  long long image_halves;        // per (problem, objective)
};

inline __host__ __device__ int round_up(int x, int r) { return (x + r - 1) / r * r; }

// Outcome transforms applied before Standardize (Sec. 5.2 S4): per objective
// a 3-bit code, code & 3 = 0 identity, 1 log (latency), 2 logit (quality);
// code & 4 negates (a maximised outcome becomes a minimised one). Several
// objectives' codes are packed 3 bits apiece, objective t at bit 3t.
inline __host__ __device__ int objective_code(int codes, int t) { return (codes >> (3 * t)) & 7; }
#ifdef __CUDACC__
// (out of line: the transforms' fp64 logarithm stays out of the kernels'
// register allocation; the identity costs a test)
static __device__ __noinline__ double outcome_transform_call(double y, int code) {
  double v = y;
  if ((code & 3) == 1) v = log(y);
  else if ((code & 3) == 2) v = log(y / (1.0 - y));
  return (code & 4) ? -v : v;
}
__device__ __forceinline__ double outcome_transform(double y, int code) {
  return code ? outcome_transform_call(y, code) : y;
}
#endif

// The side input's coordinates and inverse lengthscales carry a constant
// factor: x / l times sqrt(5) / ln 2 (the Matern-5/2 kernel, and the composite
// kernel's routing features), sqrt(3) / ln 2 on the composite kernel's
// deployment features (its Matern-3/2 part). The scaled distance r' then is
// the kernel's exponent in base 2, exp(-sqrt5 r) = 2^(-r'), with no rounding
// of a product in between.
constexpr double kCoordScale52 = 3.225964182229561;   // sqrt(5) / ln 2
constexpr double kCoordScale32 = 2.4988211106473432;  // sqrt(3) / ln 2

// Floats of one training-point chunk of the posterior's side input: X/ls as
// fp32 hi [DP][32] and lo [DP][32] (dimension-major, so pairs of training
// points load as packed f32x2), alpha as an fp32 pair, hi [32] and lo [32],
// then the objective's parameters 1/ls hi [DP], 1/ls lo [DP], and 8 scalars
// (kParS2 .. below).
inline __host__ __device__ int xt_chunk_floats(int DP) {
  return 2 * BOUTE_KCHUNK * DP + 2 * BOUTE_KCHUNK + 2 * DP + 8;
}
inline __host__ __device__ int xt_alpha_offset(int DP) { return 2 * BOUTE_KCHUNK * DP; }
inline __host__ __device__ int xt_param_offset(int DP) {
  return 2 * BOUTE_KCHUNK * DP + 2 * BOUTE_KCHUNK;
}
// The scalars after 1/ls hi and lo: outputscale; the composite kernel's s2_c,
// s2_x and d_tau; the power-of-two exponent e_W of W's operand scale; the
// composite kernel's largest training-point preference weight (written by the
// fit, in chunk 0 only).
// With in-sample draws, chunk 0 also holds the exponents of H's and G's
// operand scales (written by the in-sample preparation).
enum { kParS2 = 0, kParS2c = 1, kParS2x = 2, kParDtau = 3, kParEW = 4, kParWmax = 5, kParEH = 6,
       kParEG = 7 };

// Operand scales. The contraction runs on fp16 hi/lo parts, whose normal
// range is [2^-14, 65504]: K* is scaled by 2^e_r so that its bound lies in
// [2^14, 2^15), and W by 2^e_W with |W| <= 1/sigma_n (the smallest eigenvalue
// of K = K0 + sigma_n^2 I is at least sigma_n^2, so ||L^-1||_2 <= 1/sigma_n)
// mapped below 2^14, leaving a factor 4 of headroom for the rounding of the
// fp32 factor. Powers of two scale exactly; the epilogue divides the sum of
// squares by 2^(2 (e_r + e_W)).
inline __host__ __device__ int kstar_scale_exp(float bound) { return 14 - ilogbf(bound); }
inline __host__ __device__ int w_scale_exp(double noise, double s2) {
  // (noise floored at 1e-12 s2: a smaller noise leaves K numerically singular in fp32)
  const double v = noise > 1e-12 * s2 ? noise : 1e-12 * s2;
  return 13 - ilogb(1.0 / sqrt(v));
}

// S_in > 0: the in-sample draws' blocks after W's (a noisy acquisition's
// posterior, Sec. 5.2): H^T (n rows) and G^T (S_in rows), dense, every chunk.
inline PostPlan make_post_plan(int n, int S_in = 0) {
  PostPlan p{};
  p.n = n;
  p.npad = round_up(n, BOUTE_KCHUNK);
  p.nxt = round_up(n, BOUTE_ACHUNK) / BOUTE_KCHUNK;
  p.nchunk = p.nxt / 2;
  p.nwblk = (n + BOUTE_BLKCOLS - 1) / BOUTE_BLKCOLS;
  p.nhblk = S_in > 0 ? p.nwblk : 0;
  p.S_in = S_in > 0 ? S_in : 0;
  p.nblk = p.nwblk + p.nhblk + (p.S_in + BOUTE_BLKCOLS - 1) / BOUTE_BLKCOLS;
  long long off = 0;
  for (int q = 0; q < p.nblk; ++q) {
    const bool wq = q < p.nwblk;
    // rows of this block: W and H^T have n, G^T has S_in
    const int c0 = BOUTE_BLKCOLS * (wq ? q : q < p.nwblk + p.nhblk ? q - p.nwblk
                                                                      : q - p.nwblk - p.nhblk);
    const int rows = q < p.nwblk + p.nhblk ? n : p.S_in;
    const int w = rows - c0 < BOUTE_BLKCOLS ? rows - c0 : BOUTE_BLKCOLS;
    p.ncol[q] = round_up(w, 16);
    // W's rows < c0 + w need columns < c0 + w; the dense blocks need them all
    p.kc[q] = wq ? (c0 + w + BOUTE_ACHUNK - 1) / BOUTE_ACHUNK : p.nchunk;
    p.off[q] = off;
    off += (long long)p.kc[q] * 2 * p.ncol[q] * BOUTE_ACHUNK;
  }
  p.image_halves = off;
  return p;
}

// Half offset, inside a [rows x 64] fp16 block laid out for a K-major
// tcgen05 operand with the 128-byte swizzle, of element (row, kk): each row
// is 128 B, its 16-byte groups of 8 halves permuted by XOR with (row mod 8).
inline __host__ __device__ int sw128_off16(int row, int kk) {
  return row * 64 + ((((kk >> 3) ^ (row & 7))) << 3) + (kk & 7);
}

#ifdef __CUDACC__
// ---------------------------------------------------------------- device only
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// One plain arrival (release semantics at CTA scope for the calling thread).
__device__ __forceinline__ void mbar_arrive_count(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t phase) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(phase)
      : "memory");
  return ok != 0;
}

// As mbar_try_wait, but the thread may stay suspended in hardware for up to
// hint_ns while the phase is incomplete (it resumes as soon as the phase
// completes), so a waiting warp takes no issue slots from the working ones.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t phase,
                                                    uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(phase), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

// Waits for the given phase parity; gives up after limit_ns and returns
// false so the caller can record BOUTE_ERR_TIMEOUT instead of hanging.
__device__ __forceinline__ bool mbar_wait_ns(uint64_t *bar, uint32_t phase, uint64_t limit_ns) {
  if (mbar_try_wait(bar, phase)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, phase)) return true;
    if ((it & 63) == 0 && globaltimer() - t0 > limit_ns) return false;
  }
}
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t phase) {
  return mbar_wait_ns(bar, phase, BOUTE_WAIT_NS);
}

// Bulk copy global -> shared through the TMA engine; completion is counted
// on bar in bytes. dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Bulk copy shared -> global through the TMA engine, tracked by this
// thread's bulk groups (bulk_commit / bulk_wait_read / bulk_wait). src, dst
// 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_s2g(void *dst, const void *src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
               "r"(smem_u32(src)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// the sources of all this thread's committed bulk stores have been read
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// all this thread's committed bulk stores are complete
__device__ __forceinline__ void bulk_wait() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// Expected transaction bytes without an arrival, and an arrival counted
// `count` times (an mbarrier whose phase needs both).
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive_n(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(count)
               : "memory");
}

// Named CTA barrier `id` (1..15; 0 is __syncthreads) over `count` threads, a
// multiple of 32; every warp taking part calls it the same number of times.
__device__ __forceinline__ void named_barrier_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// ---- programmatic dependent launch -----------------------------------------------
// A kernel launched with programmatic stream serialization may start while its
// predecessor in the stream is still running: it must call pdl_wait() before
// reading anything that predecessor writes. pdl_trigger() lets the successor
// start launching; without it the successor launches when this grid's blocks
// have exited. Both are no-ops for a grid launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---- tcgen05 (5th-generation tensor cores, tensor memory) -------------------
__device__ __forceinline__ void tmem_alloc(uint32_t *dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row
// atoms of 128 B stacked contiguously (stride 1024 B).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);  // start address
  d |= (uint64_t)1 << 16;                   // leading byte offset (unused with this swizzle)
  d |= (uint64_t)(1024 >> 4) << 32;         // stride byte offset
  d |= (uint64_t)1 << 46;                   // descriptor version
  d |= (uint64_t)2 << 61;                   // 128-byte swizzle
  return d;
}

// Instruction descriptor: kind::f16 with fp16 A and B, fp32 accumulate, A
// and B K-major, M = 128, N = n (a multiple of 16, at most 256).
__host__ __device__ constexpr uint32_t idesc_f16(int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(BOUTE_TILE_M >> 4) << 24);
}

// D (tensor memory) += A (shared) x B (shared)^T, or D = A x B^T when
// accumulate is 0; issued by one thread.
__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                        uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// 32 lanes x 32 bit, 8 consecutive columns per thread; the wait is fused so
// the registers cannot be consumed early.
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, float (&v)[8]) {
  uint32_t r[8];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7])::"memory");
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}

// Two fp32 values as packed fp16 (round to nearest even): element `a` in the
// low half (the lower address in memory), `b` in the high half.
__device__ __forceinline__ uint32_t pack_f16x2(float a, float b) {
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(b), "f"(a));
  return r;
}
__device__ __forceinline__ void unpack_f16x2(uint32_t v, float &a, float &b) {
  asm("{\n\t.reg .b16 l, h;\n\tmov.b32 {l, h}, %2;\n\t"
      "cvt.f32.f16 %0, l;\n\tcvt.f32.f16 %1, h;\n\t}"
      : "=f"(a), "=f"(b)
      : "r"(v));
}
// The fp16 hi/lo split of a pair: hi = fp16(x), lo = fp16(x - hi), so that
// hi + lo carries 22 significant bits of x (x within the fp16 normal range).
__device__ __forceinline__ void split_f16x2(float x0, float x1, uint32_t &hi, uint32_t &lo) {
  hi = pack_f16x2(x0, x1);
  float h0, h1;
  unpack_f16x2(hi, h0, h1);
  lo = pack_f16x2(x0 - h0, x1 - h1);
}

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
__device__ __forceinline__ unsigned long long f2_add(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ unsigned long long f2_mul(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ unsigned long long f2_pack(float x, float y) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
  return r;
}
__device__ __forceinline__ void f2_split(unsigned long long v, float &x, float &y) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(v));
}

// 2^k as an fp32 value, k in the normal range [-126, 127].
__device__ __forceinline__ float exp2i(int k) { return __int_as_float((127 + k) << 23); }

__device__ __forceinline__ void set_status(int *status, int code) {
  if (status) atomicCAS(status, 0, code);
}
#endif

}  // namespace boute
