// Device helpers shared by the CUDA translation units of libboute:
// bounded mbarrier waits, bulk (TMA-engine) copies, tcgen05 tensor-core and
// tensor-memory wrappers, and the operand-image layout that the fit writes and
// the posterior kernel reads. sm_103a only.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "boute.h"

#define BOUTE_MAX_D 32       // candidate dimension limit (registers per thread)
#define BOUTE_MAX_M 4        // objectives per problem
#define BOUTE_MAX_N 2048     // training points per problem
#define BOUTE_MAX_PASS 12    // 256-column passes of the posterior contraction
#define BOUTE_TILE_M 128     // candidates per posterior tile (MMA M)
#define BOUTE_KCHUNK 32      // reduction columns per operand chunk (128 B of fp32)
#define BOUTE_WAIT_NS 2000000000ull  // bound on any single device-side wait

namespace boute {

// ---------------------------------------------------------------- host/device
// Operand-image plan of the posterior contraction for one (problem, objective):
// output columns [0, n) are the rows of L^-1, padded with zero rows to a
// multiple of 16. Columns are processed in passes of at most 256 (one
// tcgen05.mma N); pass p needs the reduction chunks [0, kc[p]) only, because
// row j of L^-1 is zero beyond column j. (The mean K* alpha is reduced on the
// CUDA cores while K* is built, in compensated fp32.)
struct PostPlan {
  int n, npad, ncols, npass, nchunk;
  int col0[BOUTE_MAX_PASS], ncol[BOUTE_MAX_PASS], kc[BOUTE_MAX_PASS];
  long long off[BOUTE_MAX_PASS];  // float offset of the pass's first chunk image
  long long image_floats;         // per (problem, objective)
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

// Floats of one training-point chunk of the posterior's side input: X/ls as
// fp32 hi [DP][32] and lo [DP][32] (dimension-major, so pairs of training
// points load as packed f32x2), alpha [32], then the objective's parameters
// 1/ls hi [DP], 1/ls lo [DP], outputscale, 3 floats of padding.
inline __host__ __device__ int xt_chunk_floats(int DP) {
  return 2 * BOUTE_KCHUNK * DP + BOUTE_KCHUNK + 2 * DP + 4;
}
inline __host__ __device__ int xt_param_offset(int DP) { return 2 * BOUTE_KCHUNK * DP + BOUTE_KCHUNK; }

inline PostPlan make_post_plan(int n) {
  PostPlan p{};
  p.n = n;
  p.npad = round_up(n, BOUTE_KCHUNK);
  p.nchunk = p.npad / BOUTE_KCHUNK;
  p.ncols = round_up(n, 16);
  p.npass = (p.ncols + 255) / 256;
  long long off = 0;
  for (int q = 0; q < p.npass; ++q) {
    p.col0[q] = 256 * q;
    p.ncol[q] = (p.ncols - p.col0[q]) < 256 ? (p.ncols - p.col0[q]) : 256;
    const int last_col = p.col0[q] + p.ncol[q] - 1;
    const int need = round_up(last_col + 1, BOUTE_KCHUNK);
    p.kc[q] = (need < p.npad ? need : p.npad) / BOUTE_KCHUNK;
    p.off[q] = off;
    off += (long long)p.kc[q] * 2 * p.ncol[q] * BOUTE_KCHUNK;
  }
  p.image_floats = off;
  return p;
}

// Float offset, inside a [rows x 32] fp32 block laid out for a K-major
// tcgen05 operand with the 128-byte swizzle, of element (row, kk): each row
// is 128 B, 16-byte groups permuted by XOR with (row mod 8).
inline __host__ __device__ int sw128_off(int row, int kk) {
  return row * 32 + ((((kk >> 2) ^ (row & 7))) << 2) + (kk & 3);
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

// Instruction descriptor: kind::tf32, fp32 accumulate, A and B K-major, M=128.
__host__ __device__ constexpr uint32_t idesc_tf32(int N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(BOUTE_TILE_M >> 4) << 24);
}

__device__ __forceinline__ void mma_tf32(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
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

// Round to the nearest tf32 value (ties away), kept in fp32 layout.
__device__ __forceinline__ float tf32_rna(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

__device__ __forceinline__ void set_status(int *status, int code) {
  if (status) atomicCAS(status, 0, code);
}
#endif

}  // namespace boute
