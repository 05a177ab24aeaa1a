// Gradient coding with cyclic repetition (GC-CR) on the device, for the naive
// pipelined construction of §V-A and for GC-CR itself:
//
//   gc_encoding_kernel  worker j's encoding coefficients c_{j,l} (its row of
//                       B, supported on partitions j..j+s mod n) from the
//                       construction's random matrix H (s x n, H 1 = 0):
//                       c_{j,0} = 1 and the other s solve
//                       H[:, {j+1..j+s}] x = -H[:, j], so H B[j]^T = 0.
//                       Once per run.
//   gc_weights_kernel   the step's decode weights d(J) with
//                       sum_m d_m B[j_m] = 1 over the received workers J,
//                       the per-(worker, slot) weights d_j c_{j,l} / n the
//                       decode applies, and the range of the decoding
//                       coefficients alpha_{m,k} = d_m c_{j_m,l}.  Per step.
//   gc_decode_kernel    ghat = sum over received j and slots l of
//                       (d_j c_{j,l} / n) * store[j][l] (slot l of worker j
//                       holds its latest gradient of D_{(j+l) mod n}), then
//                       beta <- beta - eta ghat (§III).
//
// Both solves are Gaussian elimination with partial pivoting in fp64 by one
// warp (n <= kGcMaxN, so each lane owns at most two rows).  A pivot below
// kGcPivotTol times the largest coefficient, or a decode system whose
// solution misses sum_m d_m B[j_m] = 1 by more than kGcResidTol (relative),
// sets kErrSingular: those draws cannot encode, or that straggler set cannot
// be decoded.
#include "tail.cuh"

namespace pgc {

namespace {

constexpr double kGcPivotTol = 1e-13;
constexpr double kGcResidTol = 1e-8;
constexpr int kGcLd = kGcMaxN + 1;   // leading dimension of the augmented systems

__device__ __forceinline__ double warp_max_f64(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ double warp_sum_f64(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Solve the rows x cols system M[:, 0:cols] x = M[:, cols] (row-major, leading
// dimension kGcLd, rows >= cols, rows <= 64) in place by one warp: lane l owns
// rows l and l + 32.  Pivot rows are chosen per column by largest magnitude
// among the rows not used yet (no rows move; piv[] records the order); rows
// left over after cols pivots are not used (the caller checks consistency).
// Writes x[0:cols] (shared) and returns false on a singular pivot.
__device__ bool warp_solve(double* M, int rows, int cols, double* x, int* piv) {
  const int lane = threadIdx.x & 31;
  bool used0 = lane >= rows, used1 = lane + 32 >= rows;
  double scale = 0.0;
  for (int r = lane; r < rows; r += 32)
    for (int q = 0; q < cols; ++q) scale = fmax(scale, fabs(M[r * kGcLd + q]));
  scale = warp_max_f64(scale);
  for (int k = 0; k < cols; ++k) {
    // pivot: the unused row with the largest |M[r][k]|; ties to the lower row
    double bv = -1.0;
    int br = rows;
    if (!used0) { bv = fabs(M[lane * kGcLd + k]); br = lane; }
    if (!used1) {
      const double v = fabs(M[(lane + 32) * kGcLd + k]);
      if (v > bv) { bv = v; br = lane + 32; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const double ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int orr = __shfl_xor_sync(0xffffffffu, br, o);
      if (ov > bv || (ov == bv && orr < br)) { bv = ov; br = orr; }
    }
    if (!(bv > kGcPivotTol * scale)) return false;
    const int p = br;
    if (lane == 0) piv[k] = p;
    if (p == lane) used0 = true;
    if (p == lane + 32) used1 = true;
    __syncwarp();
    const double* Mp = M + p * kGcLd;
    const double inv = 1.0 / Mp[k];
    for (int h = 0; h < 2; ++h) {
      const int r = lane + 32 * h;
      if (h == 0 ? used0 : used1) continue;
      double* Mr = M + r * kGcLd;
      const double f = Mr[k] * inv;
      for (int q = k + 1; q <= cols; ++q) Mr[q] = fma(-f, Mp[q], Mr[q]);
      Mr[k] = 0.0;
    }
    __syncwarp();
  }
  // back-substitution in pivot order; lanes split the inner sum
  for (int k = cols - 1; k >= 0; --k) {
    const double* Mp = M + piv[k] * kGcLd;
    double acc = 0.0;
    for (int q = k + 1 + lane; q < cols; q += 32) acc = fma(Mp[q], x[q], acc);
    acc = warp_sum_f64(acc);
    if (lane == 0) x[k] = (Mp[cols] - acc) / Mp[k];
    __syncwarp();
  }
  return true;
}

// Entry (r, col) of H = [draws | -(row sums of draws)].
__device__ __forceinline__ double h_entry(const double* draws, int n, int r, int col, const double* rowsum) {
  return col < n - 1 ? draws[(int64_t)r * (n - 1) + col] : -rowsum[r];
}

}  // namespace

// grid n (one warp per worker j), block 32.  coeff: [n][c], c = s + 1.
__global__ void __launch_bounds__(32) gc_encoding_kernel(const double* __restrict__ draws, int n, int s,
                                                         double* __restrict__ coeff, int* status) {
  __shared__ double M[kGcMaxN * kGcLd];
  __shared__ double rowsum[kGcMaxN];
  __shared__ double x[kGcMaxN];
  __shared__ int piv[kGcMaxN];
  const int j = blockIdx.x, lane = threadIdx.x;
  const int c = s + 1;
  for (int r = lane; r < s; r += 32) {
    double t = 0.0;
    for (int q = 0; q < n - 1; ++q) t += draws[(int64_t)r * (n - 1) + q];
    rowsum[r] = t;
  }
  __syncwarp();
  // M = [H[:, j+1..j+s] | -H[:, j]], s x (s + 1)
  for (int r = lane; r < s; r += 32) {
    for (int q = 0; q < s; ++q) M[r * kGcLd + q] = h_entry(draws, n, r, (j + 1 + q) % n, rowsum);
    M[r * kGcLd + s] = -h_entry(draws, n, r, j, rowsum);
  }
  __syncwarp();
  const bool ok = s == 0 || warp_solve(M, s, s, x, piv);
  if (!ok) {
    if (lane == 0) atomicOr(status, kErrSingular);
    return;
  }
  for (int l = lane; l < c; l += 32) coeff[(int64_t)j * c + l] = l == 0 ? 1.0 : x[l - 1];
}

// grid 1, block 32.  Outputs: d [n] (0 for stragglers), wts [n][c] fp32
// d_j c_{j,l} / n, coeff_out [n] fp32 d_j / n (the per-worker coefficient of
// the coded gradient), alpha [2] = max, min of d_j c_{j,l} over received j.
__global__ void __launch_bounds__(32) gc_weights_kernel(GcWeightsArgs a) {
  __shared__ double M[kGcMaxN * kGcLd];
  __shared__ double x[kGcMaxN];
  __shared__ int piv[kGcMaxN];
  __shared__ int recv[kGcMaxN];
  const int lane = threadIdx.x;
  const int n = a.n, c = a.c;
  // the received workers, ascending
  int nr = 0;
  for (int base = 0; base < n; base += 32) {
    const int i = base + lane;
    const bool rc = i < n && !((a.mask.w[i >> 5] >> (i & 31)) & 1u);
    const unsigned bal = __ballot_sync(0xffffffffu, rc);
    if (rc) recv[nr + __popc(bal & ((1u << lane) - 1u))] = i;
    nr += __popc(bal);
  }
  __syncwarp();
  if (nr != n - a.s) {
    for (int q = lane; q < n * c; q += 32) a.wts[q] = 0.f;
    if (lane == 0) atomicOr(a.status, kErrBadMask);
    return;
  }
  // M[k][m] = B[j_m][k] (n x nr), right-hand side 1
  for (int k = lane; k < n; k += 32) {
    for (int m = 0; m < nr; ++m) {
      const int l = (k - recv[m] + n) % n;
      M[k * kGcLd + m] = l < c ? a.coeff[(int64_t)recv[m] * c + l] : 0.0;
    }
    M[k * kGcLd + nr] = 1.0;
  }
  __syncwarp();
  bool ok = warp_solve(M, n, nr, x, piv);
  // consistency: every partition's decoding coefficients must sum to 1
  if (ok) {
    double res = 0.0, xmax = 0.0, bmax = 0.0;
    for (int k = lane; k < n; k += 32) {
      double t = 0.0;
      for (int m = 0; m < nr; ++m) {
        const int l = (k - recv[m] + n) % n;
        if (l < c) {
          const double b = a.coeff[(int64_t)recv[m] * c + l];
          t = fma(x[m], b, t);
          bmax = fmax(bmax, fabs(b));
        }
      }
      res = fmax(res, fabs(t - 1.0));
    }
    for (int m = lane; m < nr; m += 32) xmax = fmax(xmax, fabs(x[m]));
    res = warp_max_f64(res);
    xmax = warp_max_f64(xmax);
    bmax = warp_max_f64(bmax);
    ok = res <= kGcResidTol * (1.0 + xmax * bmax);
  }
  if (!ok) {
    // no weights: the decode leaves beta unchanged and the host reports the error
    for (int q = lane; q < n * c; q += 32) a.wts[q] = 0.f;
    if (lane == 0) atomicOr(a.status, kErrSingular);
    return;
  }
  const double inv_n = 1.0 / (double)n;
  for (int i = lane; i < n; i += 32) {
    a.d[i] = 0.0;
    a.coeff_out[i] = 0.f;
    for (int l = 0; l < c; ++l) a.wts[(int64_t)i * c + l] = 0.f;
  }
  __syncwarp();
  double amax = -INFINITY, amin = INFINITY;
  for (int m = lane; m < nr; m += 32) {
    const int j = recv[m];
    const double dj = x[m];
    a.d[j] = dj;
    a.coeff_out[j] = (float)(dj * inv_n);
    for (int l = 0; l < c; ++l) {
      const double al = dj * a.coeff[(int64_t)j * c + l];
      amax = fmax(amax, al);
      amin = fmin(amin, al);
      a.wts[(int64_t)j * c + l] = (float)(al * inv_n);
    }
  }
  amax = warp_max_f64(amax);
  amin = -warp_max_f64(-amin);
  if (lane == 0) {
    a.alpha[0] = amax;
    a.alpha[1] = amin;
  }
}

// One float4 column per thread, grid-stride; the received (worker, slot)
// weights are compacted into shared memory in (worker, slot) order and each
// column's sum issues eight loads at a time.
__global__ void __launch_bounds__(256) gc_decode_kernel(DecodeArgs a, const float* __restrict__ wts) {
  __shared__ int qi[kGcMaxN * kGcMaxN];
  __shared__ float qw[kGcMaxN * kGcMaxN];
  __shared__ int qn;
  grid_dep_launch();
  grid_dep_wait();
  const int nw = a.n * a.c;
  if (threadIdx.x < 32) {
    int cnt = 0;
    for (int base = 0; base < nw; base += 32) {
      const int q = base + threadIdx.x;
      const float v = q < nw ? __ldcg(wts + q) : 0.f;
      const bool nz = v != 0.f;
      const unsigned bal = __ballot_sync(0xffffffffu, nz);
      if (nz) {
        const int pos = cnt + __popc(bal & ((1u << threadIdx.x) - 1u));
        qi[pos] = q;          // store index = worker * c + slot
        qw[pos] = v;
      }
      cnt += __popc(bal);
    }
    if (threadIdx.x == 0) qn = cnt;
  }
  __syncthreads();
  const int cnt = qn;
  const int64_t P4 = a.P / 4;
  const float4* store = reinterpret_cast<const float4*>(a.store);
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P4; p += (int64_t)gridDim.x * blockDim.x) {
    float4 g = f4zero();
    for (int j0 = 0; j0 < cnt; j0 += 8) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = j0 + u < cnt ? __ldcg(store + (int64_t)qi[j0 + u] * P4 + p) : f4zero();
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (j0 + u < cnt) g = f4fma(qw[j0 + u], v[u], g);
    }
    float4 w = __ldcg(reinterpret_cast<const float4*>(a.w) + p);
    w = f4fma(-a.lr, g, w);
    store_outputs(a, p, g, w);
  }
}

cudaError_t launch_gc_encoding(const double* draws, int n, int s, double* coeff, int* status, cudaStream_t st) {
  if (n < 1 || n > kGcMaxN || s < 0 || s >= n) return cudaErrorInvalidValue;
  gc_encoding_kernel<<<n, 32, 0, st>>>(draws, n, s, coeff, status);
  return cudaGetLastError();
}

cudaError_t launch_gc_decode(const GcWeightsArgs& w, const DecodeArgs& a, cudaStream_t st, bool pdl, int sm_count) {
  if (a.n < 1 || a.n > kGcMaxN || a.c < 1 || a.c > a.n) return cudaErrorInvalidValue;
  gc_weights_kernel<<<1, 32, 0, st>>>(w);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int64_t blocks = (a.P / 4 + 255) / 256;
  if (blocks > (int64_t)sm_count * 8) blocks = (int64_t)sm_count * 8;
  if (blocks < 1) blocks = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gc_decode_kernel, a, static_cast<const float*>(w.wts));
}

}  // namespace pgc
