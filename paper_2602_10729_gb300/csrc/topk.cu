// Deterministic top-k per problem. Values become 64-bit keys (order-preserving
// float bits in the high word, the complement of the index in the low word), so
// one unsigned comparison orders by value descending, then index ascending.
// k <= 32 takes a warp-register path in one launch (below). Otherwise, level 1: every block sorts one segment of kSeg keys in shared memory
// (bitonic) and keeps its k largest. Further levels apply the same segment
// sort to the surviving keys until one segment per problem remains; the last
// level writes indices and values. All levels are fully parallel across
// blocks; nothing waits on another block.
#include <math.h>

#include <algorithm>

#include "internal.h"
#include "warp_select.cuh"

namespace boute {

namespace {

constexpr int kThreads = 512;
constexpr int kSeg = 2048;  // keys per segment (16 KB of shared memory)

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
  pdl_wait();
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
      if (BOUTE_INB(i, k) && BOUTE_INB(j, N)) {
        idx[(size_t)b * k + i] = (long long)j;
        val[(size_t)b * k + i] = acq[(size_t)b * N + j];
      }
    }
  } else {
    unsigned long long *out = keys_out + ((size_t)b * nseg + seg) * k;
    for (int i = threadIdx.x; i < k; i += blockDim.x) out[i] = i < L ? buf[i] : 0ull;
  }
}

// ---- k <= 32: one warp holds a running top 32, one key per lane ----------------
// Lane i holds the i-th largest key seen so far. A batch of 32 new keys is
// rejected with one ballot when none beats the current 32nd; otherwise it is
// sorted across the lanes (bitonic network on shuffles) and merged: the
// element-wise maximum of the running list and the reversed batch is a bitonic
// sequence holding the 32 largest keys of both, which five more shuffle steps
// sort. Each block merges its warps' lists; a second launch merges the blocks'.
constexpr int kWarpBlock = 256;  // threads; 8 warps
constexpr int kWarpBatches = 8;  // batches of 32 keys a warp loads at once

// Block blockIdx.x of problem blockIdx.y takes entries [x * per_block,
// (x+1) * per_block) of the problem's N values and forms their 32 largest
// keys. With one block per problem it writes the final k indices and values.
// Otherwise each block stores its 32 keys in `keys` and counts itself done on
// the problem's counter; the block that finishes last merges all the blocks'
// lists (eight warps, then one) and writes the result, and sets the counter
// back to zero for the next call.
__global__ void __launch_bounds__(kWarpBlock) warp_topk_kernel(
    const float *vals, long long N, long long per_block, unsigned long long *keys,
    unsigned *counter, int k, long long *idx, float *val) {
  __shared__ unsigned long long lists[kWarpBlock / 32][kWarpK];
  __shared__ int is_last;
  pdl_wait();
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int G = gridDim.x;
  const long long lo = (long long)blockIdx.x * per_block;
  const long long hi = std::min<long long>(N, lo + per_block);
  const size_t row = (size_t)b * N;
  unsigned long long top = 0ull;  // below every real key
  for (long long base = lo + (long long)warp * 32 * kWarpBatches; base < hi;
       base += (long long)kWarpBlock * kWarpBatches) {
    unsigned long long x[kWarpBatches];
#pragma unroll
    for (int u = 0; u < kWarpBatches; ++u) {
      const long long g = base + 32 * u + lane;
      x[u] = g < hi ? make_key(__ldcs(vals + row + g), (unsigned)g) : 0ull;
    }
#pragma unroll
    for (int u = 0; u < kWarpBatches; ++u) {
      const unsigned long long thr = shfl64(top, 31);
      if (__ballot_sync(0xffffffffu, x[u] > thr) == 0u) continue;
      top = warp_merge_desc(top, warp_sort_desc(x[u], lane), lane);
    }
  }
  lists[warp][lane] = top;
  __syncthreads();
  if (warp == 0) {
#pragma unroll 1
    for (int w = 1; w < kWarpBlock / 32; ++w) top = warp_merge_desc(top, lists[w][lane], lane);
    if (G > 1) {
      keys[((size_t)b * G + blockIdx.x) * kWarpK + lane] = top;
      __threadfence();  // the list is visible before the block counts itself done
      __syncwarp();
      if (lane == 0) is_last = atomicAdd(&counter[b], 1u) == (unsigned)(G - 1);
    }
  }
  if (G > 1) {
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    top = 0ull;
    for (int l = warp; l < G; l += kWarpBlock / 32)
      top = warp_merge_desc(top, __ldcg(keys + ((size_t)b * G + l) * kWarpK + lane), lane);
    lists[warp][lane] = top;
    __syncthreads();
    if (warp != 0) return;
#pragma unroll 1
    for (int w = 1; w < kWarpBlock / 32; ++w) top = warp_merge_desc(top, lists[w][lane], lane);
    if (lane == 0) counter[b] = 0u;
  } else if (warp != 0) {
    return;
  }
  if (lane < k) {
    const unsigned j = key_index(top);
    if (BOUTE_INB(lane, k)) {
      idx[(size_t)b * k + lane] = (long long)j;
      val[(size_t)b * k + lane] = vals[row + j];
    }
  }
}

// scratch: B x G x 32 keys, then B counters (zero on entry, zero on exit)
int launch_topk_warp(const float *acq, int B, long long N, int k, long long *idx, float *val,
                     void *scratch, bool counters_zeroed, cudaStream_t s) {
  // at most 256 first-level blocks per problem, each a multiple of 2048 entries
  const long long unit = (long long)kWarpBlock * kWarpBatches;
  long long per_block = unit;
  while ((N + per_block - 1) / per_block > 256) per_block += unit;
  const long long G = (N + per_block - 1) / per_block;
  prefer_shared(warp_topk_kernel);
  unsigned long long *keys = G > 1 ? (unsigned long long *)scratch : nullptr;
  unsigned *counter = G > 1 ? (unsigned *)(keys + (size_t)B * G * kWarpK) : nullptr;
  if (G > 1 && !counters_zeroed && cudaMemsetAsync(counter, 0, B * sizeof(unsigned), s) != cudaSuccess)
    return last_launch_status();
  launch_pdl(warp_topk_kernel, dim3((unsigned)G, B), dim3(kWarpBlock), 0, s, acq, N, per_block,
             keys, counter, k, idx, val);
  count_launch(1);
  return last_launch_status();
}

}  // namespace

// Scratch for the levels after the first: two ping-pong key arrays of
// ceil(N / 2048) * k keys per problem (segment path), or at most
// ceil(N / 2048) runs of 32 keys per problem and one counter per problem
// (warp path, k <= 32); k is counted as at least 32 so that one bound covers
// both.
size_t topk_scratch_bytes(int B, long long N, int k) {
  const long long g1 = (N + kSeg - 1) / kSeg;
  if (g1 <= 1) return 16;
  return 2 * (size_t)B * g1 * std::max(k, 32) * sizeof(unsigned long long) + 16;
}

int launch_topk(const float *acq, int B, long long N, int k, long long *idx, float *val,
                void *scratch, cudaStream_t s, bool counters_zeroed) {
  if (k > kSeg / 2) return BOUTE_ERR_UNSUPPORTED;
  if (k <= kWarpK)
    return launch_topk_warp(acq, B, N, k, idx, val, scratch, counters_zeroed, s);
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

BOUTE_BOUNDS_READER(topk)

}  // namespace boute
