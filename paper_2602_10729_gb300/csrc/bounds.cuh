// Bounds checks of the debug build. Compiled with BOUTE_DEBUG_BOUNDS, every
// BOUTE_INB(index, extent) tests 0 <= index < extent; the first index out of
// its extent in a translation unit is recorded (its source line, the index,
// the extent) and the guarded access is skipped, so that a wrong index shows
// up as a report (boute_bounds_report) instead of a fault. In the product
// library the checks compile to `true` and cost nothing.
//
// Each translation unit that includes this header and uses the checks keeps
// its own record (no relocatable device code) and defines its reader with
// BOUTE_BOUNDS_READER(name); the C-ABI collects them.
#pragma once

#include <cuda_runtime.h>

namespace boute {

struct BoundsRecord {
  unsigned long long flag;  // 1 once an index has been out of its extent
  long long line, index, extent;
};

#ifdef BOUTE_DEBUG_BOUNDS
static __device__ BoundsRecord g_bounds_record;

__device__ __forceinline__ bool bounds_ok(long long index, long long extent, int line) {
  if (index >= 0 && index < extent) return true;
  if (atomicCAS(&g_bounds_record.flag, 0ull, 1ull) == 0ull) {
    g_bounds_record.line = line;
    g_bounds_record.index = index;
    g_bounds_record.extent = extent;
  }
  return false;
}
#define BOUTE_INB(index, extent) \
  ::boute::bounds_ok((long long)(index), (long long)(extent), __LINE__)
// Reader of this translation unit's record: copies it to `out` (4 words:
// flag, line, index, extent) and clears it.
#define BOUTE_BOUNDS_READER(name)                                                        \
  int bounds_read_##name(long long *out) {                                               \
    BoundsRecord r{};                                                                    \
    if (cudaMemcpyFromSymbol(&r, g_bounds_record, sizeof(r)) != cudaSuccess) return -1;  \
    const BoundsRecord z{};                                                              \
    if (cudaMemcpyToSymbol(g_bounds_record, &z, sizeof(z)) != cudaSuccess) return -1;    \
    out[0] = (long long)r.flag;                                                          \
    out[1] = r.line;                                                                     \
    out[2] = r.index;                                                                    \
    out[3] = r.extent;                                                                   \
    return 0;                                                                            \
  }
#else
#define BOUTE_INB(index, extent) true
#define BOUTE_BOUNDS_READER(name) \
  int bounds_read_##name(long long *out) {  \
    out[0] = out[1] = out[2] = out[3] = 0;  \
    return 0;                               \
  }
#endif

}  // namespace boute
