// Deterministic top-k per problem. Values become 64-bit keys (order-preserving
// float bits in the high word, the complement of the index in the low word), so
// one unsigned comparison orders by value descending, then index ascending.
// Level 1: every block sorts one segment of kSeg keys in shared memory
// (bitonic) and keeps its k largest. Further levels apply the same segment
// sort to the surviving keys until one segment per problem remains; the last
// level writes indices and values. All levels are fully parallel across
// blocks; nothing waits on another block.
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace boute {

namespace {

constexpr int kThreads = 512;
constexpr int kSeg = 2048;  // keys per segment (16 KB of shared memory)

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

// Sort buf[0, L) descending, L a power of two.
__device__ void bitonic_desc(unsigned long long *buf, int L) {
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
}

// One segment of problem b: keys [seg*kSeg, seg*kSeg + kSeg) of a row of
// `len` entries (values when FROM_VALUES, else keys). Keeps the k largest.
template <bool FROM_VALUES>
__global__ void __launch_bounds__(kThreads) segment_topk_kernel(
    const float *vals, const unsigned long long *keys_in, long long len, int k, int nseg,
    unsigned long long *keys_out, const float *acq, long long N, long long *idx, float *val) {
  __shared__ unsigned long long buf[kSeg];
  const int b = blockIdx.y, seg = blockIdx.x;
  const long long base = (long long)seg * kSeg;
  const long long n_here = std::min<long long>(kSeg, len - base);
  int L = 2;
  while (L < n_here) L <<= 1;
  for (int i = threadIdx.x; i < L; i += blockDim.x) {
    unsigned long long key = 0ull;  // below every real key
    if (i < n_here) {
      const long long g = base + i;
      key = FROM_VALUES ? make_key(__ldcs(vals + (size_t)b * len + g), (unsigned)g)
                        : keys_in[(size_t)b * len + g];
    }
    buf[i] = key;
  }
  __syncthreads();
  bitonic_desc(buf, L);
  if (idx) {  // final level: one segment per problem
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
      const unsigned j = key_index(buf[i]);
      idx[(size_t)b * k + i] = (long long)j;
      val[(size_t)b * k + i] = acq[(size_t)b * N + j];
    }
  } else {
    unsigned long long *out = keys_out + ((size_t)b * nseg + seg) * k;
    for (int i = threadIdx.x; i < k; i += blockDim.x) out[i] = i < L ? buf[i] : 0ull;
  }
}

}  // namespace

// Scratch for the levels after the first: two ping-pong key arrays.
size_t topk_scratch_bytes(int B, long long N, int k) {
  const long long g1 = (N + kSeg - 1) / kSeg;
  if (g1 <= 1) return 16;
  return 2 * (size_t)B * g1 * k * sizeof(unsigned long long) + 16;
}

int launch_topk(const float *acq, int B, long long N, int k, long long *idx, float *val,
                void *scratch, cudaStream_t s) {
  if (k > kSeg / 2) return BOUTE_ERR_UNSUPPORTED;
  long long len = N;
  long long nseg = (len + kSeg - 1) / kSeg;
  unsigned long long *ping = (unsigned long long *)scratch;
  unsigned long long *pong = ping + (size_t)B * nseg * k;
  int launches = 0;
  if (nseg == 1) {
    segment_topk_kernel<true><<<dim3(1, B), kThreads, 0, s>>>(acq, nullptr, len, k, 1, nullptr,
                                                              acq, N, idx, val);
    count_launch(1);
    return last_launch_status();
  }
  segment_topk_kernel<true><<<dim3((unsigned)nseg, B), kThreads, 0, s>>>(
      acq, nullptr, len, k, (int)nseg, ping, acq, N, nullptr, nullptr);
  ++launches;
  len = nseg * k;
  for (;;) {
    nseg = (len + kSeg - 1) / kSeg;
    if (nseg == 1) {
      segment_topk_kernel<false><<<dim3(1, B), kThreads, 0, s>>>(nullptr, ping, len, k, 1,
                                                                 nullptr, acq, N, idx, val);
      ++launches;
      break;
    }
    segment_topk_kernel<false><<<dim3((unsigned)nseg, B), kThreads, 0, s>>>(
        nullptr, ping, len, k, (int)nseg, pong, acq, N, nullptr, nullptr);
    ++launches;
    std::swap(ping, pong);
    len = nseg * k;
  }
  count_launch(launches);
  return last_launch_status();
}

}  // namespace boute
