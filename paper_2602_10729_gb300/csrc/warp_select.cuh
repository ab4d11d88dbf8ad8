// Selection keys and warp-register top-32 lists, shared by the top-k kernels
// and the acquisition kernels that select as they score.
//
// A key orders candidates by value descending, then index ascending, in one
// unsigned comparison: order-preserving float bits (NaN as -infinity, -0 as
// +0) in the high word, the complement of the index in the low word. A warp
// list holds 32 keys, one per lane, sorted descending (lane 0 the largest).
#pragma once

#include <cuda_runtime.h>
#include <math.h>

namespace boute {

constexpr int kWarpK = 32;

__device__ __forceinline__ unsigned long long make_key(float v, unsigned idx) {
  if (isnan(v)) v = -INFINITY;
  if (v == 0.f) v = 0.f;  // -0 sorts as +0
  unsigned u = __float_as_uint(v);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)u << 32) | (unsigned long long)(0xFFFFFFFFu - idx);
}

__device__ __forceinline__ unsigned key_index(unsigned long long key) {
  return 0xFFFFFFFFu - (unsigned)(key & 0xFFFFFFFFull);
}

__device__ __forceinline__ unsigned long long shfl64(unsigned long long v, int src) {
  return __shfl_sync(0xffffffffu, v, src);
}
__device__ __forceinline__ unsigned long long shfl_xor64(unsigned long long v, int m) {
  return __shfl_xor_sync(0xffffffffu, v, m);
}

// Sort one key per lane, descending across the lanes.
__device__ __forceinline__ unsigned long long warp_sort_desc(unsigned long long x, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const unsigned long long y = shfl_xor64(x, stride);
      const bool desc = (lane & size) == 0 || size == 32;
      const bool lower = (lane & stride) == 0;
      const unsigned long long mx = x > y ? x : y, mn = x > y ? y : x;
      x = (lower == desc) ? mx : mn;
    }
  }
  return x;
}

// top, s: descending across the lanes. Returns the 32 largest of both, descending.
__device__ __forceinline__ unsigned long long warp_merge_desc(unsigned long long top,
                                                              unsigned long long s, int lane) {
  const unsigned long long r = shfl64(s, 31 - lane);
  unsigned long long u = top > r ? top : r;
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) {
    const unsigned long long y = shfl_xor64(u, stride);
    const bool lower = (lane & stride) == 0;
    u = lower ? (u > y ? u : y) : (u > y ? y : u);
  }
  return u;
}

// Insert one key (the same in every lane) into a sorted warp list.
__device__ __forceinline__ unsigned long long warp_insert_desc(unsigned long long top,
                                                               unsigned long long key, int lane) {
  const int pos = __popc(__ballot_sync(0xffffffffu, top > key));  // keys above the new one
  const unsigned long long up = __shfl_up_sync(0xffffffffu, top, 1);
  return lane < pos ? top : (lane == pos ? key : up);
}

// A warp's running top-32 fed one key at a time (the same key in every lane):
// keys wait in a lane each (lane i holds the i-th since the last merge) and
// are sorted and merged into the list 32 at a time, so that adding a key
// costs a select. flush() merges what is pending; top then holds the 32
// largest keys added, descending (zero where fewer were added).
struct WarpTopBatch {
  unsigned long long top = 0ull, pend = 0ull;
  int count = 0;  // pending keys (the same in every lane)
  __device__ __forceinline__ void add(unsigned long long key, int lane) {
    if (lane == count) pend = key;
    if (++count == kWarpK) flush(lane);
  }
  __device__ __forceinline__ void flush(int lane) {
    if (count == 0) return;
    top = warp_merge_desc(top, warp_sort_desc(pend, lane), lane);
    pend = 0ull;
    count = 0;
  }
};

// Counts a block in on *p at GPU scope with acquire-release order. Release:
// what this thread wrote, or observed before a barrier it passed, is visible
// to whoever observes the new count. Acquire: a thread that observes the
// final count sees all of that, and so does its block after a barrier.
__device__ __forceinline__ unsigned atomic_add_acq_rel_gpu(unsigned *p, unsigned v) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// Merge the lists of a block's 16 warps (each warp's `top`) into warp 0's
// `top` as a tree of four levels: at level h, warps [h, 2h) hand their lists
// to warps [0, h) through `lists`. Every thread of the block must call it;
// the caller synchronises before `lists` is written again.
__device__ __forceinline__ unsigned long long block_merge16(unsigned long long (*lists)[kWarpK],
                                                           unsigned long long top, int warp,
                                                           int lane) {
#pragma unroll
  for (int h = 8; h >= 1; h >>= 1) {
    if (warp >= h && warp < 2 * h) lists[warp][lane] = top;
    __syncthreads();
    if (warp < h) top = warp_merge_desc(top, lists[warp + h][lane], lane);
  }
  return top;
}

}  // namespace boute
