// Top-k selection whose level-to-level scratch is a fixed, statically
// allocated device array instead of memory taken from the CUDA pool. The
// selection itself is the same launch sequence as boute_select_topk; only the
// place the intermediate keys live differs.
#include <cuda_runtime.h>

#include <mutex>

#include "internal.h"

namespace boute {

namespace {

// Scratch of the levels after the first: two ping-pong arrays of 64-bit keys.
// The only words that must start at zero (one counter per problem, on the
// k <= 32 path) are cleared by every call before its kernel runs; every key
// is written before it is read.
static __device__ __align__(256) unsigned char g_topk_scratch[BOUTE_TOPK_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
void *g_scratch_ptr[kMaxDevices] = {};
std::mutex g_scratch_mu;

// Address of the current device's copy of the array, looked up once per device.
int scratch_address(void **out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return BOUTE_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_topk_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return BOUTE_ERR_CUDA;
    }
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return BOUTE_OK;
}

}  // namespace

}  // namespace boute

using namespace boute;

extern "C" int boute_select_topk_noalloc(const float *acq, int B, long long N, int k,
                                         long long *idx, float *val, void *stream) {
  BOUTE_TRACE();
  if (!acq || !idx || !val || B < 1 || N < 1 || k < 1 || k > 1024 || k > N)
    return BOUTE_ERR_INVALID_ARG;
  if ((long long)B * N >= (1ll << 31)) return BOUTE_ERR_INVALID_ARG;
  const long long nseg = (N + 2047) / 2048;  // first-level segments per problem
  const unsigned long long need =
      nseg <= 1 ? 0ull
                : 2ull * (unsigned long long)B * nseg * (k < 32 ? 32 : k) * sizeof(unsigned long long);
  if (need > BOUTE_TOPK_NOALLOC_SCRATCH_BYTES) return BOUTE_ERR_UNSUPPORTED;
  if (int r = device_ok()) return r;
  void *scratch = nullptr;
  if (int r = scratch_address(&scratch)) return r;
  return launch_topk(acq, B, N, k, idx, val, scratch, (cudaStream_t)stream);
}
