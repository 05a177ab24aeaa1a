// Softmax cross-entropy partition gradient on CUDA cores, any K (§III with
// f = log sum_k exp(w_k.x) - w_y.x):
//   Z = X_e W^T            (tiled fp32 FMA, features widened from bf16/fp32)
//   R = softmax(Z) - onehot(y)      (row-wise, in place)
//   partial[e] = R^T X_e   ([K][ld], unscaled; the commit applies 1/m_e)
// Also provides the tiled logits pass used by the full-loss kernel.
#include "dev_common.cuh"
#include "pgc_internal.h"
#include "pgc.h"

namespace pgc {

constexpr int TB = 64;     // tile edge (rows x classes, or classes x features)
constexpr int TK = 16;     // reduction chunk

template <typename T>
__device__ __forceinline__ float ldx(const T* p);
template <>
__device__ __forceinline__ float ldx<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ldx<uint16_t>(const uint16_t* p) { return bf16_bits_to_float(*p); }

// Z[zrow0 + r][k] = sum_j X[row0 + r][j] W[k][j]  for r < rows, k < K.
// grid: (ceil(K / 64), ceil(max_rows / 64), nE); 256 threads, 4x4 outputs each.
template <typename T>
__global__ void __launch_bounds__(256) logits_tiled(const T* __restrict__ X, int64_t ld, const float* __restrict__ W,
                                                    int64_t K, const int64_t* e_row0, const int64_t* e_rows,
                                                    const int64_t* e_zrow0, float* __restrict__ Z, int64_t Kpad) {
  const int e = blockIdx.z;
  const int64_t rows = e_rows[e];
  const int64_t r0 = (int64_t)blockIdx.y * TB;
  const int64_t k0 = (int64_t)blockIdx.x * TB;
  if (r0 >= rows) return;
  const T* Xe = X + e_row0[e] * ld;
  __shared__ float xs[TK][TB + 4];
  __shared__ float ws[TK][TB + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int64_t j0 = 0; j0 < ld; j0 += TK) {
    for (int q = threadIdx.x; q < TB * TK; q += 256) {
      const int rr = q / TK, jj = q % TK;
      const int64_t r = r0 + rr, k = k0 + rr, j = j0 + jj;
      xs[jj][rr] = (r < rows && j < ld) ? ldx<T>(Xe + r * ld + j) : 0.f;
      ws[jj][rr] = (k < K && j < ld) ? W[k * ld + j] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int jj = 0; jj < TK; ++jj) {
      float xv[4], wv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { xv[i] = xs[jj][ty * 4 + i]; wv[i] = ws[jj][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[i][q] = fmaf(xv[i], wv[q], acc[i][q]);
    }
    __syncthreads();
  }
  const int64_t zr0 = e_zrow0[e];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = r0 + ty * 4 + i;
    if (r >= rows) continue;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t k = k0 + tx * 4 + q;
      if (k < K) Z[(zr0 + r) * Kpad + k] = acc[i][q];
    }
  }
}

// R = softmax(Z) - onehot(y), one warp per row, in place.
__global__ void softmax_residual(float* __restrict__ Z, int64_t Kpad, int64_t K, const int32_t* __restrict__ y,
                                 const int64_t* e_row0, const int64_t* e_rows, const int64_t* e_zrow0, int nE,
                                 int64_t total) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t zr = warp; zr < total; zr += nwarps) {
    // find the partition of this Z row (nE is small; linear scan)
    int e = 0;
    while (e + 1 < nE && e_zrow0[e + 1] <= zr) ++e;
    const int64_t grow = e_row0[e] + (zr - e_zrow0[e]);
    float* z = Z + zr * Kpad;
    float m = -INFINITY;
    for (int64_t k = lane; k < K; k += 32) m = fmaxf(m, z[k]);
    m = warp_max(m);
    float sum = 0.f;
    for (int64_t k = lane; k < K; k += 32) sum += expf(z[k] - m);
    sum = warp_sum(sum);
    const float inv = 1.0f / sum;
    const int lab = y[grow];
    for (int64_t k = lane; k < K; k += 32) z[k] = expf(z[k] - m) * inv - (k == lab ? 1.0f : 0.0f);
  }
}

// partial[e][k * ld + j] = sum_{r < rows_e} R[zrow0 + r][k] * X[row0 + r][j]
// grid: (ceil(ld / 64), ceil(K / 64), nE)
template <typename T>
__global__ void __launch_bounds__(256) backward_tiled(const T* __restrict__ X, int64_t ld, const float* __restrict__ Z,
                                                      int64_t Kpad, int64_t K, const int64_t* e_row0,
                                                      const int64_t* e_rows, const int64_t* e_zrow0,
                                                      float* __restrict__ partials) {
  const int e = blockIdx.z;
  const int64_t rows = e_rows[e];
  const int64_t j0 = (int64_t)blockIdx.x * TB;
  const int64_t k0 = (int64_t)blockIdx.y * TB;
  const T* Xe = X + e_row0[e] * ld;
  const float* Ze = Z + e_zrow0[e] * Kpad;
  __shared__ float rs[TK][TB + 4];
  __shared__ float xs[TK][TB + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int64_t r0 = 0; r0 < rows; r0 += TK) {
    for (int q = threadIdx.x; q < TB * TK; q += 256) {
      const int rr = q / TB, cc = q % TB;
      const int64_t r = r0 + rr;
      const int64_t k = k0 + cc, j = j0 + cc;
      rs[rr][cc] = (r < rows && k < K) ? Ze[r * Kpad + k] : 0.f;
      xs[rr][cc] = (r < rows && j < ld) ? ldx<T>(Xe + r * ld + j) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int rr = 0; rr < TK; ++rr) {
      float rv[4], xv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { rv[i] = rs[rr][ty * 4 + i]; xv[i] = xs[rr][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[i][q] = fmaf(rv[i], xv[q], acc[i][q]);
    }
    __syncthreads();
  }
  float* out = partials + (int64_t)e * K * ld;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t k = k0 + ty * 4 + i;
    if (k >= K) continue;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t j = j0 + tx * 4 + q;
      if (j < ld) out[k * ld + j] = acc[i][q];
    }
  }
}

// R = softmax(Z) - onehot(y) written as bf16 for the tensor-core backward;
// one warp per row of an evaluated partition, zero for the padded classes.
// R = softmax(Z) - onehot(y) in bf16 for one row per warp, the row held in
// registers: lane l owns the float4 columns l, l + 32, ... (NV per lane, the
// padded class count is 128 NV).  Classes K..Kpad-1 and the rows up to the
// next multiple of 64 (the backward GEMM's K padding) are written as zeros,
// since another phase may have left values there.  The grid also zeroes
// zero_buf (the slot total that the backward GEMM accumulates into).
template <int NV>
__global__ void __launch_bounds__(256) softmax_residual_bf16(const float* __restrict__ Z, uint16_t* __restrict__ Rb,
                                                             int64_t K, const int32_t* __restrict__ y,
                                                             const int64_t* e_row0, const int64_t* e_rows,
                                                             const int64_t* e_zrow0, float* zero_buf, int64_t zero_n4) {
  constexpr int64_t Kpad = 128 * NV;
  const int e = blockIdx.y;
  if (zero_buf) {
    const int64_t nthr = (int64_t)gridDim.x * gridDim.y * blockDim.x;
    const int64_t tid = ((int64_t)blockIdx.y * gridDim.x + blockIdx.x) * blockDim.x + threadIdx.x;
    for (int64_t i = tid; i < zero_n4; i += nthr) reinterpret_cast<float4*>(zero_buf)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  const int lane = threadIdx.x & 31;
  const int64_t rows = e_rows[e];
  const int64_t rows_pad = (rows + 63) / 64 * 64;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r = warp; r < rows_pad; r += nwarps) {
    const int64_t zr = e_zrow0[e] + r;
    uint2* out = reinterpret_cast<uint2*>(Rb + zr * Kpad);
    if (r >= rows) {
#pragma unroll
      for (int j = 0; j < NV; ++j) out[lane + 32 * j] = make_uint2(0u, 0u);
      continue;
    }
    const float4* z4 = reinterpret_cast<const float4*>(Z + zr * Kpad);
    float4 v[NV];
#pragma unroll
    for (int j = 0; j < NV; ++j) v[j] = __ldcs(z4 + lane + 32 * j);   // read once: streaming
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int64_t k0 = 4 * (lane + 32 * j);
      if (k0 + 0 < K) m = fmaxf(m, v[j].x);
      if (k0 + 1 < K) m = fmaxf(m, v[j].y);
      if (k0 + 2 < K) m = fmaxf(m, v[j].z);
      if (k0 + 3 < K) m = fmaxf(m, v[j].w);
    }
    m = warp_max(m);
    float sum = 0.f;
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int64_t k0 = 4 * (lane + 32 * j);
      v[j].x = k0 + 0 < K ? expf(v[j].x - m) : 0.f;
      v[j].y = k0 + 1 < K ? expf(v[j].y - m) : 0.f;
      v[j].z = k0 + 2 < K ? expf(v[j].z - m) : 0.f;
      v[j].w = k0 + 3 < K ? expf(v[j].w - m) : 0.f;
      sum += (v[j].x + v[j].y) + (v[j].z + v[j].w);
    }
    sum = warp_sum(sum);
    const float inv = 1.0f / sum;
    const int lab = y[e_row0[e] + r];
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int64_t k0 = 4 * (lane + 32 * j);
      const float r0 = v[j].x * inv - (k0 + 0 == lab ? 1.f : 0.f);
      const float r1 = v[j].y * inv - (k0 + 1 == lab ? 1.f : 0.f);
      const float r2 = v[j].z * inv - (k0 + 2 == lab ? 1.f : 0.f);
      const float r3 = v[j].w * inv - (k0 + 3 == lab ? 1.f : 0.f);
      __nv_bfloat162 lo = __floats2bfloat162_rn(k0 + 0 < K ? r0 : 0.f, k0 + 1 < K ? r1 : 0.f);
      __nv_bfloat162 hi = __floats2bfloat162_rn(k0 + 2 < K ? r2 : 0.f, k0 + 3 < K ? r3 : 0.f);
      out[lane + 32 * j] = make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
    }
  }
}

cudaError_t launch_softmax_bf16(const float* Z, uint16_t* Rb, int64_t Kpad, int64_t K, const int32_t* y,
                                const int64_t* e_row0, const int64_t* e_rows, const int64_t* e_zrow0, int nE,
                                int64_t max_rows, float* zero_buf, int64_t zero_n, cudaStream_t st) {
  if (nE <= 0) return cudaSuccess;
  // about four rows per warp, and at least a few CTAs per partition
  int64_t warps = ((max_rows + 63) / 64 * 64 + 3) / 4;
  int64_t bx = (warps + 7) / 8;
  if (bx < 4) bx = 4;
  if (bx > 1024) bx = 1024;
  const dim3 grid((unsigned)bx, (unsigned)nE);
  const int64_t n4 = zero_n / 4;
  switch (Kpad) {
    case 256: softmax_residual_bf16<2><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 512: softmax_residual_bf16<4><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 768: softmax_residual_bf16<6><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 1024: softmax_residual_bf16<8><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 1280: softmax_residual_bf16<10><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 1536: softmax_residual_bf16<12><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 1792: softmax_residual_bf16<14><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    case 2048: softmax_residual_bf16<16><<<grid, 256, 0, st>>>(Z, Rb, K, y, e_row0, e_rows, e_zrow0, zero_buf, n4); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_softmax_cc(const SoftmaxCCArgs& a, cudaStream_t st) {
  if (a.nE <= 0) return cudaSuccess;
  const dim3 g1((unsigned)((a.K + TB - 1) / TB), (unsigned)((a.max_rows + TB - 1) / TB), (unsigned)a.nE);
  if (a.dtype == PGC_BF16)
    logits_tiled<uint16_t><<<g1, 256, 0, st>>>(static_cast<const uint16_t*>(a.X), a.ld, a.W, a.K, a.e_row0,
                                                a.e_rows, a.e_zrow0, a.Z, a.Kpad);
  else
    logits_tiled<float><<<g1, 256, 0, st>>>(static_cast<const float*>(a.X), a.ld, a.W, a.K, a.e_row0, a.e_rows,
                                             a.e_zrow0, a.Z, a.Kpad);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  // total Z rows = zrow0 of the last partition + its rows; computed by the host
  softmax_residual<<<1024, 256, 0, st>>>(a.Z, a.Kpad, a.K, a.y, a.e_row0, a.e_rows, a.e_zrow0, a.nE, a.z_total);
  err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  const dim3 g3((unsigned)((a.ld + TB - 1) / TB), (unsigned)((a.K + TB - 1) / TB), (unsigned)a.nE);
  if (a.dtype == PGC_BF16)
    backward_tiled<uint16_t><<<g3, 256, 0, st>>>(static_cast<const uint16_t*>(a.X), a.ld, a.Z, a.Kpad, a.K,
                                                  a.e_row0, a.e_rows, a.e_zrow0, a.partials);
  else
    backward_tiled<float><<<g3, 256, 0, st>>>(static_cast<const float*>(a.X), a.ld, a.Z, a.Kpad, a.K, a.e_row0,
                                               a.e_rows, a.e_zrow0, a.partials);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Full loss F(beta) = (1 / rows) sum f (§III), fp64 accumulation.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void loss_rows_kernel(LossArgs a) {
  __shared__ double red[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const T* X = static_cast<const T*>(a.X);
  const float* y = static_cast<const float*>(a.y);
  double acc = 0.0;
  for (int64_t r = warp; r < a.rows; r += nwarps) {
    float dot = 0.f;
    for (int64_t j = lane; j < a.ld; j += 32) dot = fmaf(ldx<T>(X + r * a.ld + j), a.w[j], dot);
    dot = warp_sum(dot);
    if (lane == 0) {
      const double z = dot, yy = y[r];
      const double f = a.loss == PGC_LOGISTIC ? (fmax(z, 0.0) + log1p(exp(-fabs(z))) - yy * z)
                                              : 0.5 * (z - yy) * (z - yy);
      acc += f;
    }
  }
  if (lane == 0) red[wid] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
    a.blocksum[blockIdx.x] = s;
  }
}

// per-row softmax loss from a chunk of logits Z[rows][Kpad]
__global__ void loss_softmax_rows(const float* __restrict__ Z, int64_t Kpad, int64_t K, const int32_t* __restrict__ y,
                                  int64_t row0, int64_t rows, double* blocksum) {
  __shared__ double red[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  double acc = 0.0;
  for (int64_t r = warp; r < rows; r += nwarps) {
    const float* z = Z + r * Kpad;
    float m = -INFINITY;
    for (int64_t k = lane; k < K; k += 32) m = fmaxf(m, z[k]);
    m = warp_max(m);
    float s = 0.f;
    for (int64_t k = lane; k < K; k += 32) s += expf(z[k] - m);
    s = warp_sum(s);
    if (lane == 0) acc += (double)m + log((double)s) - (double)z[y[row0 + r]];
  }
  if (lane == 0) red[wid] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t += red[i];
    blocksum[blockIdx.x] += t;
  }
}

__global__ void loss_finish(const double* blocksum, int nblocks, int64_t rows, double* out) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    double s = 0.0;
    for (int i = 0; i < nblocks; ++i) s += blocksum[i];
    *out = s / (double)rows;
  }
}

__global__ void zero_doubles(double* p, int n) {
  for (int i = threadIdx.x; i < n; i += blockDim.x) p[i] = 0.0;
}

cudaError_t launch_loss(const LossArgs& a, cudaStream_t st) {
  if (a.loss != PGC_SOFTMAX) {
    if (a.dtype == PGC_BF16) loss_rows_kernel<uint16_t><<<a.nblocks, 256, 0, st>>>(a);
    else loss_rows_kernel<float><<<a.nblocks, 256, 0, st>>>(a);
  } else {
    // logits in chunks of rows (bounded scratch), then per-row loss; chunk i
    // is described on the device by {row0, rows, 0} at chunk_desc[3 i]
    zero_doubles<<<1, 256, 0, st>>>(a.blocksum, a.nblocks);
    const int64_t chunk = a.z_chunk_rows;
    for (int64_t r0 = 0, i = 0; r0 < a.rows; r0 += chunk, ++i) {
      const int64_t rows = a.rows - r0 < chunk ? a.rows - r0 : chunk;
      const dim3 g((unsigned)((a.K + TB - 1) / TB), (unsigned)((rows + TB - 1) / TB), 1);
      const int64_t* desc = a.chunk_desc + 3 * i;
      if (a.dtype == PGC_BF16)
        logits_tiled<uint16_t><<<g, 256, 0, st>>>(static_cast<const uint16_t*>(a.X), a.ld, a.w, a.K, desc,
                                                   desc + 1, desc + 2, a.Z, a.Kpad);
      else
        logits_tiled<float><<<g, 256, 0, st>>>(static_cast<const float*>(a.X), a.ld, a.w, a.K, desc, desc + 1,
                                                desc + 2, a.Z, a.Kpad);
      loss_softmax_rows<<<a.nblocks, 256, 0, st>>>(a.Z, a.Kpad, a.K, static_cast<const int32_t*>(a.y), r0, rows,
                                                   a.blocksum);
      const cudaError_t e = cudaGetLastError();
      if (e != cudaSuccess) return e;
    }
  }
  loss_finish<<<1, 32, 0, st>>>(a.blocksum, a.nblocks, a.rows, a.out);
  return cudaGetLastError();
}

}  // namespace pgc
