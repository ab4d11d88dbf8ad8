// Deterministic top-k per problem. Values become 64-bit keys (order-preserving
// float bits in the high word, the complement of the index in the low word), so
// one unsigned comparison orders by value descending, then index ascending.
// Phase 1: G blocks per problem stream their segment, keep a running top-k in
// shared memory and append only keys above the running k-th key; the buffer
// is bitonic-sorted when it fills. Phase 2: one block per problem merges the
// G partial lists the same way.
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace boute {

namespace {

constexpr int kThreads = 512;
constexpr int kBuf = 4096;  // keys in shared memory (32 KB)
constexpr long long kSegment = 16384;

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

// Sort buf[0, cnt) descending (pads to a power of two with 0, the smallest key),
// then keep the first k. Returns the new count; updates the threshold.
__device__ int flush(unsigned long long *buf, int cnt, int k, unsigned long long *thresh) {
  int L = 2;
  while (L < cnt) L <<= 1;
  for (int i = cnt + threadIdx.x; i < L; i += blockDim.x) buf[i] = 0ull;
  __syncthreads();
  for (int size = 2; size <= L; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (L >> 1); i += blockDim.x) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const unsigned long long x = buf[lo], y = buf[hi];
        if ((x < y) == desc && x != y) {
          buf[lo] = y;
          buf[hi] = x;
        }
      }
      __syncthreads();
    }
  }
  const int kept = cnt < k ? cnt : k;
  if (threadIdx.x == 0 && kept == k) *thresh = buf[k - 1];
  __syncthreads();
  return kept;
}

template <bool FROM_KEYS>
__device__ void stream_topk(const float *vals, const unsigned long long *keys, long long begin,
                            long long end, int k, unsigned long long *buf, int *s_add,
                            unsigned long long *s_thresh, int &cnt) {
  for (long long base = begin; base < end; base += blockDim.x) {
    if (cnt + (int)blockDim.x > kBuf) cnt = flush(buf, cnt, k, s_thresh);
    const unsigned long long th = *s_thresh;
    const long long i = base + threadIdx.x;
    if (i < end) {
      const unsigned long long key = FROM_KEYS ? keys[i] : make_key(__ldcs(vals + i), (unsigned)i);
      if (key > th) buf[cnt + atomicAdd(s_add, 1)] = key;
    }
    __syncthreads();
    cnt += *s_add;
    __syncthreads();
    if (threadIdx.x == 0) *s_add = 0;
    __syncthreads();
  }
}

__global__ void __launch_bounds__(kThreads) topk_partial_kernel(const float *acq, long long N,
                                                                int k, int G,
                                                                unsigned long long *part) {
  __shared__ unsigned long long buf[kBuf];
  __shared__ int s_add;
  __shared__ unsigned long long s_thresh;
  const int b = blockIdx.y, g = blockIdx.x;
  const long long len = (N + G - 1) / G;
  const long long begin = std::min<long long>(N, (long long)g * len);
  const long long end = std::min<long long>(N, begin + len);
  if (threadIdx.x == 0) {
    s_add = 0;
    s_thresh = 0ull;
  }
  __syncthreads();
  int cnt = 0;
  stream_topk<false>(acq + (size_t)b * N, nullptr, begin, end, k, buf, &s_add, &s_thresh, cnt);
  cnt = flush(buf, cnt, k, &s_thresh);
  unsigned long long *out = part + ((size_t)b * G + g) * k;
  for (int i = threadIdx.x; i < k; i += blockDim.x) out[i] = i < cnt ? buf[i] : 0ull;
}

__global__ void __launch_bounds__(kThreads) topk_merge_kernel(const unsigned long long *part,
                                                              int G, int k, const float *acq,
                                                              long long N, long long *idx,
                                                              float *val) {
  __shared__ unsigned long long buf[kBuf];
  __shared__ int s_add;
  __shared__ unsigned long long s_thresh;
  const int b = blockIdx.x;
  if (threadIdx.x == 0) {
    s_add = 0;
    s_thresh = 0ull;
  }
  __syncthreads();
  int cnt = 0;
  stream_topk<true>(nullptr, part + (size_t)b * G * k, 0, (long long)G * k, k, buf, &s_add,
                    &s_thresh, cnt);
  cnt = flush(buf, cnt, k, &s_thresh);
  for (int i = threadIdx.x; i < k; i += blockDim.x) {
    const unsigned j = key_index(buf[i]);
    idx[(size_t)b * k + i] = (long long)j;
    val[(size_t)b * k + i] = acq[(size_t)b * N + j];
  }
}

int groups_for(int B, long long N, int k) {
  long long G = (N + kSegment - 1) / kSegment;
  G = std::min<long long>(G, 64);
  G = std::min<long long>(G, std::max<long long>(1, (long long)(4 * kBuf) / std::max(1, k)));
  return (int)std::max<long long>(1, G);
}

}  // namespace

size_t topk_scratch_bytes(int B, long long N, int k) {
  return (size_t)B * groups_for(B, N, k) * k * sizeof(unsigned long long);
}

int launch_topk(const float *acq, int B, long long N, int k, long long *idx, float *val,
                void *scratch, cudaStream_t s) {
  const int G = groups_for(B, N, k);
  topk_partial_kernel<<<dim3(G, B), kThreads, 0, s>>>(acq, N, k, G,
                                                      (unsigned long long *)scratch);
  topk_merge_kernel<<<B, kThreads, 0, s>>>((const unsigned long long *)scratch, G, k, acq, N,
                                           idx, val);
  count_launch(2);
  return last_launch_status();
}

}  // namespace boute
