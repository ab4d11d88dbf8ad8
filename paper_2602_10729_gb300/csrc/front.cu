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

__global__ void pareto_kernel(const double *Ys, int n, int m, const double *ref,
                              unsigned char *mask, double *front, int *P) {
  extern __shared__ long long yk[];  // n*m keys, then n keep flags (as int)
  int *keep = (int *)(yk + (size_t)n * m);
  __shared__ int count;
  __shared__ long long rk[BOUTE_MAX_M];
  const int b = blockIdx.x;
  const double *Yb = Ys + (size_t)b * n * m;
  for (int e = threadIdx.x; e < n * m; e += blockDim.x) yk[e] = dkey(Yb[e]);
  if (threadIdx.x < m) rk[threadIdx.x] = dkey(ref[(size_t)b * m + threadIdx.x]);
  if (threadIdx.x == 0) count = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const long long *yi = yk + (size_t)i * m;
    bool k = true;
    for (int t = 0; t < m; ++t)
      if (!(yi[t] < rk[t])) k = false;
    for (int j = 0; j < n && k; ++j) {
      if (j == i) continue;
      const long long *yj = yk + (size_t)j * m;
      if (dominates(yj, yi, m) || (j < i && equal(yj, yi, m))) k = false;
    }
    keep[i] = k;
    mask[(size_t)b * n + i] = (unsigned char)k;
    if (k) atomicAdd(&count, 1);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    if (!keep[i]) continue;
    const long long *yi = yk + (size_t)i * m;
    int rank = 0;
    for (int j = 0; j < n; ++j)
      if (keep[j] && lex_less(yk + (size_t)j * m, j, yi, i, m)) ++rank;
    double *dst = front + ((size_t)b * n + rank) * m;
    for (int t = 0; t < m; ++t) dst[t] = Yb[(size_t)i * m + t];
  }
  if (threadIdx.x == 0) P[b] = count;
}

// ---- boxes ---------------------------------------------------------------------
// m = 2: strip i = [a_i, b_i) x (-inf, u_i) of the staircase (P+1 strips).
// m = 3: sweep the front by increasing f3; between consecutive levels the
// cross-section of the improving region is the 2-D staircase region of the
// points below the level. Each strip lives from the level where it appears to
// the level where an inserted point changes it, and becomes one box
// [a, b) x (-inf, u) x [z_birth, z_death); every insertion creates at most two
// strips, so there are at most 2P+1 boxes.
__global__ void boxes_kernel(const double *front, const int *P, int n, int m, const double *ref,
                             float *lower, float *upper, int *Kout) {
  extern __shared__ double ws[];
  const int b = blockIdx.x, cap = 2 * n + 2;
  const int Pb = P[b];
  const double *F = front + (size_t)b * n * m;
  const double *r = ref + (size_t)b * m;
  float *lo = lower + (size_t)b * cap * m, *hi = upper + (size_t)b * cap * m;
  if (m == 2) {
    for (int i = threadIdx.x; i <= Pb; i += blockDim.x) {
      lo[2 * i] = i == 0 ? -INFINITY : (float)F[2 * (i - 1)];
      lo[2 * i + 1] = -INFINITY;
      hi[2 * i] = i == Pb ? (float)r[0] : (float)F[2 * i];
      hi[2 * i + 1] = i == 0 ? (float)r[1] : (float)F[2 * (i - 1) + 1];
    }
    if (threadIdx.x == 0) Kout[b] = Pb + 1;
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
    if (z1 > z0 && bb > a && K < cap) {
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
  Kout[b] = K;
}

}  // namespace

int launch_pareto(const double *Ys, int B, int n, int m, const double *ref, unsigned char *mask,
                  double *front, int *P, cudaStream_t s) {
  const size_t smem = (size_t)n * m * sizeof(long long) + (size_t)n * sizeof(int);
  if (smem > 48 * 1024)
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
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(boxes_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  boxes_kernel<<<B, 256, smem, s>>>(front, P, n, m, ref, lower, upper, K);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
