// Pareto front of the observed (standardised) outcomes and the disjoint box
// decomposition of the region that improves on it. One block per problem;
// fronts are small (tens of points), the work is O(n^2) compares.
#include <math.h>

#include "internal.h"

namespace boute {

namespace {

// Order-preserving integer image of a double (-0 taken as +0): x < y exactly
// when key(x) < key(y), for finite values. Comparing keys keeps the O(n^2)
// dominance tests on the integer pipes instead of the slow fp64 unit.
__device__ __forceinline__ long long dkey(double x) {
  if (x == 0.0) x = 0.0;
  const long long b = __double_as_longlong(x);
  return b >= 0 ? b : (long long)(b ^ 0x7FFFFFFFFFFFFFFFll);
}

// a dominates b (minimisation): <= everywhere, < somewhere
__device__ __forceinline__ bool dominates(const long long *a, const long long *b, int m) {
  bool lt = false;
  for (int t = 0; t < m; ++t) {
    if (a[t] > b[t]) return false;
    if (a[t] < b[t]) lt = true;
  }
  return lt;
}

__device__ __forceinline__ bool equal(const long long *a, const long long *b, int m) {
  for (int t = 0; t < m; ++t)
    if (a[t] != b[t]) return false;
  return true;
}

// (Y_j, j) < (Y_i, i) lexicographically
__device__ __forceinline__ bool lex_less(const long long *yj, int j, const long long *yi, int i,
                                         int m) {
  for (int t = 0; t < m; ++t) {
    if (yj[t] < yi[t]) return true;
    if (yj[t] > yi[t]) return false;
  }
  return j < i;
}

// All ordered pairs (i, j) are spread over the block's threads: a point is
// dropped as soon as one pair shows it dominated (or a duplicate of a smaller
// index), and its rank among the kept points is a count over pairs too.
// smem: n*m keys, n drop flags, n ranks. Writes mask, front rows, P.
__device__ void pareto_block(const double *Yb, int n, int m, const double *rb,
                             unsigned char *mask, double *front, int *P, void *smem) {
  long long *yk = (long long *)smem;
  int *drop = (int *)(yk + (size_t)n * m);
  int *rank = drop + n;
  __shared__ int count;
  __shared__ long long rk[BOUTE_MAX_M];
  for (int e = threadIdx.x; e < n * m; e += blockDim.x) yk[e] = dkey(Yb[e]);
  if (threadIdx.x < m) rk[threadIdx.x] = dkey(rb[threadIdx.x]);
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    drop[i] = 0;
    rank[i] = 0;
  }
  if (threadIdx.x == 0) count = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const long long *yi = yk + (size_t)i * m;
    for (int t = 0; t < m; ++t)
      if (!(yi[t] < rk[t])) drop[i] = 1;
  }
  const long long nn = (long long)n * n;
  for (long long e = threadIdx.x; e < nn; e += blockDim.x) {
    const int i = (int)(e / n), j = (int)(e % n);
    if (j == i) continue;
    const long long *yi = yk + (size_t)i * m, *yj = yk + (size_t)j * m;
    if (dominates(yj, yi, m) || (j < i && equal(yj, yi, m))) drop[i] = 1;  // benign race: all write 1
  }
  __syncthreads();
  for (long long e = threadIdx.x; e < nn; e += blockDim.x) {
    const int i = (int)(e / n), j = (int)(e % n);
    if (drop[i] || drop[j] || j == i) continue;
    if (lex_less(yk + (size_t)j * m, j, yk + (size_t)i * m, i, m)) atomicAdd(&rank[i], 1);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const bool k = !drop[i];
    mask[i] = (unsigned char)k;
    if (k) {
      atomicAdd(&count, 1);
      double *dst = front + (size_t)rank[i] * m;
      for (int t = 0; t < m; ++t) dst[t] = Yb[(size_t)i * m + t];
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *P = count;
  __syncthreads();
}

__global__ void pareto_kernel(const double *Ys, int n, int m, const double *ref,
                              unsigned char *mask, double *front, int *P) {
  extern __shared__ long long smem_keys[];
  const int b = blockIdx.x;
  pareto_block(Ys + (size_t)b * n * m, n, m, ref + (size_t)b * m, mask + (size_t)b * n,
               front + (size_t)b * n * m, P + b, smem_keys);
}

// ---- boxes ---------------------------------------------------------------------
// m = 2: strip i = [a_i, b_i) x (-inf, u_i) of the staircase (P+1 strips).
// m = 3: sweep the front by increasing f3; between consecutive levels the
// cross-section of the improving region is the 2-D staircase region of the
// points below the level. Each strip lives from the level where it appears to
// the level where an inserted point changes it, and becomes one box
// [a, b) x (-inf, u) x [z_birth, z_death); every insertion creates at most two
// strips, so there are at most 2P+1 boxes.
// One problem: F = its front (P rows), r = its reference point, lo/hi = its
// box arrays (capacity 2n+2), *Kout = box count. smem (m = 3): 10 (n+2)
// doubles and n+2 ints.
__device__ void boxes_block(const double *F, int Pb, int n, int m, const double *r, float *lo,
                            float *hi, int *Kout, void *smem) {
  double *ws = (double *)smem;
  const int cap = 2 * n + 2;
  (void)cap;  // (the debug build checks the box count against it)
  if (m == 2) {
    for (int i = threadIdx.x; i <= Pb; i += blockDim.x) {
      if (!BOUTE_INB(i, cap)) break;
      lo[2 * i] = i == 0 ? -INFINITY : (float)F[2 * (i - 1)];
      lo[2 * i + 1] = -INFINITY;
      hi[2 * i] = i == Pb ? (float)r[0] : (float)F[2 * i];
      hi[2 * i + 1] = i == 0 ? (float)r[1] : (float)F[2 * (i - 1) + 1];
    }
    if (threadIdx.x == 0) *Kout = Pb + 1;
    return;
  }
  // m == 3 --------------------------------------------------------------------
  const int L = n + 2;
  double *sx = ws, *sy = sx + L;                          // staircase (f1 asc, f2 desc)
  double *ca = sy + L, *cb = ca + L, *cu = cb + L, *cz = cu + L;  // live strips
  double *na = cz + L, *nb = na + L, *nu = nb + L, *nz = nu + L;  // next strips
  int *ord = (int *)(nz + L);
  for (int i = threadIdx.x; i < Pb; i += blockDim.x) {  // order by (f3, index)
    int rank = 0;
    const double zi = F[(size_t)i * 3 + 2];
    for (int j = 0; j < Pb; ++j) {
      const double zj = F[(size_t)j * 3 + 2];
      if (zj < zi || (zj == zi && j < i)) ++rank;
    }
    ord[rank] = i;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  int ns = 0, nc = 1, K = 0;
  ca[0] = -INFINITY; cb[0] = r[0]; cu[0] = r[1]; cz[0] = -INFINITY;
  auto emit = [&](double a, double bb, double u, double z0, double z1) {
    // (a decomposition with more than cap boxes is reported by the debug build)
    if (z1 > z0 && bb > a && BOUTE_INB(K, cap)) {
      lo[K * 3 + 0] = (float)a; lo[K * 3 + 1] = -INFINITY; lo[K * 3 + 2] = (float)z0;
      hi[K * 3 + 0] = (float)bb; hi[K * 3 + 1] = (float)u; hi[K * 3 + 2] = (float)z1;
      ++K;
    }
  };
  for (int q = 0; q < Pb; ++q) {
    const double *pq = F + (size_t)ord[q] * 3;
    const double qx = pq[0], qy = pq[1], qz = pq[2];
    bool covered = false;
    for (int s = 0; s < ns && !covered; ++s)
      if (sx[s] <= qx && sy[s] <= qy) covered = true;
    if (covered) continue;
    // new staircase: drop points q weakly dominates in 2-D, insert q in f1 order
    int w = 0, ins = -1;
    for (int s = 0; s < ns; ++s) {
      if (sx[s] >= qx && sy[s] >= qy) continue;
      if (ins < 0 && sx[s] > qx) { ins = w; na[w] = qx; nb[w] = qy; ++w; }
      na[w] = sx[s]; nb[w] = sy[s]; ++w;
    }
    if (ins < 0) { na[w] = qx; nb[w] = qy; ++w; }
    for (int s = 0; s < w; ++s) { sx[s] = na[s]; sy[s] = nb[s]; }
    ns = w;
    // strips of the new staircase; a strip identical to a live one keeps its birth
    int nn = 0, j = 0;
    for (int s = 0; s <= ns; ++s) {
      const double a = s == 0 ? -INFINITY : sx[s - 1];
      const double bb = s == ns ? r[0] : sx[s];
      const double u = s == 0 ? r[1] : sy[s - 1];
      while (j < nc && ca[j] < a) { emit(ca[j], cb[j], cu[j], cz[j], qz); ++j; }
      double z = qz;
      if (j < nc && ca[j] == a && cb[j] == bb && cu[j] == u) { z = cz[j]; ++j; }
      na[nn] = a; nb[nn] = bb; nu[nn] = u; nz[nn] = z; ++nn;
    }
    while (j < nc) { emit(ca[j], cb[j], cu[j], cz[j], qz); ++j; }
    for (int s = 0; s < nn; ++s) { ca[s] = na[s]; cb[s] = nb[s]; cu[s] = nu[s]; cz[s] = nz[s]; }
    nc = nn;
  }
  for (int j = 0; j < nc; ++j) emit(ca[j], cb[j], cu[j], cz[j], r[2]);
  *Kout = K;
}

__global__ void boxes_kernel(const double *front, const int *P, int n, int m, const double *ref,
                             float *lower, float *upper, int *Kout) {
  extern __shared__ double ws_boxes[];
  const int b = blockIdx.x, cap = 2 * n + 2;
  boxes_block(front + (size_t)b * n * m, P[b], n, m, ref + (size_t)b * m,
              lower + (size_t)b * cap * m, upper + (size_t)b * cap * m, Kout + b, ws_boxes);
}

__device__ double block_sum_d(double v, double *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double t = 0.0;
  for (int w = 0; w < nw; ++w) t += red[w];
  return t;
}

// The engine's front stage, one block per problem: standardise the m outcome
// columns, take the Pareto front, decompose the improving region into boxes.
// It depends on the raw outcomes only, so it runs beside the GP fit.
__global__ void front_fused_kernel(const double *Y, int n, int m, const double *ref, double *Ys,
                                   unsigned char *mask, double *front, int *P, float *lower,
                                   float *upper, int *Kout, int want_boxes) {
  extern __shared__ long long smem_front[];
  __shared__ double red[32];
  const int b = blockIdx.x, cap = 2 * n + 2;
  const double *Yb = Y + (size_t)b * n * m;
  double *Ysb = Ys + (size_t)b * n * m;
  for (int t = 0; t < m; ++t) {
    double s = 0.0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) s += Yb[(size_t)i * m + t];
    const double mean = block_sum_d(s, red) / n;
    double ss = 0.0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const double z = Yb[(size_t)i * m + t] - mean;
      ss += z * z;
    }
    ss = block_sum_d(ss, red);
    double sd = n > 1 ? sqrt(ss / (n - 1)) : 1.0;
    if (!(sd >= 1e-8)) sd = 1.0;
    const double isd = 1.0 / sd;
    for (int i = threadIdx.x; i < n; i += blockDim.x)
      Ysb[(size_t)i * m + t] = (Yb[(size_t)i * m + t] - mean) * isd;
  }
  __syncthreads();
  __shared__ int Pb;
  pareto_block(Ysb, n, m, ref + (size_t)b * m, mask + (size_t)b * n, front + (size_t)b * n * m,
               &Pb, smem_front);
  if (threadIdx.x == 0) P[b] = Pb;
  if (want_boxes)
    boxes_block(front + (size_t)b * n * m, Pb, n, m, ref + (size_t)b * m,
                lower + (size_t)b * cap * m, upper + (size_t)b * cap * m, Kout + b, smem_front);
}

}  // namespace

int launch_pareto(const double *Ys, int B, int n, int m, const double *ref, unsigned char *mask,
                  double *front, int *P, cudaStream_t s) {
  const size_t smem = (size_t)n * m * sizeof(long long) + 2 * (size_t)n * sizeof(int) + 16;
  cudaFuncSetAttribute(pareto_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  pareto_kernel<<<B, 512, smem, s>>>(Ys, n, m, ref, mask, front, P);
  count_launch();
  return last_launch_status();
}

int launch_boxes(const double *front, const int *P, int B, int n, int m, const double *ref,
                 float *lower, float *upper, int *K, cudaStream_t s) {
  size_t smem = 0;
  if (m == 3) smem = (size_t)10 * (n + 2) * sizeof(double) + (size_t)(n + 2) * sizeof(int);
  else if (m != 2) return BOUTE_ERR_UNSUPPORTED;
  cudaFuncSetAttribute(boxes_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  boxes_kernel<<<B, 256, smem, s>>>(front, P, n, m, ref, lower, upper, K);
  count_launch();
  return last_launch_status();
}

size_t front_smem_bytes(int n, int m) {
  const size_t pk = (size_t)n * m * sizeof(long long) + 2 * (size_t)n * sizeof(int) + 16;
  const size_t bx = m == 3 ? (size_t)10 * (n + 2) * sizeof(double) + (size_t)(n + 2) * sizeof(int) : 0;
  return pk > bx ? pk : bx;
}

int launch_front_fused(const double *Y, int B, int n, int m, const double *ref, double *Ys,
                       unsigned char *mask, double *front, int *P, float *lower, float *upper,
                       int *K, int want_boxes, cudaStream_t s) {
  const size_t smem = front_smem_bytes(n, m);
  prefer_shared(front_fused_kernel);
  // (static arrays count against the same 48 KB default: always set)
  cudaFuncSetAttribute(front_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)smem);
  front_fused_kernel<<<B, 512, smem, s>>>(Y, n, m, ref, Ys, mask, front, P, lower, upper, K,
                                          want_boxes);
  count_launch();
  return last_launch_status();
}

BOUTE_BOUNDS_READER(front)

}  // namespace boute
