// Standalone tail kernels of a step (used when the gradient kernel does not
// fuse them; see tail.cuh for the arithmetic):
//   K4 commit_kernel  one CTA column-slice per evaluated partition: the new
//                     gradient g_e = (1/m_e) * ordered sum of its partials,
//                     written into every store that keeps the copy (§VI-A).
//   K6 decode_kernel  decode coefficients derived on the device from the
//                     straggler mask (§IV-A, §V-B), decode, SGD (§III).
// Both may be launched as programmatic dependents of the previous kernel:
// they wait for it (griddepcontrol.wait) before reading its results, and the
// decode derives its coefficients (which need only the mask) before waiting.
#include "tail.cuh"

namespace pgc {

// One CTA per (column slice, evaluated partition); a thread sums one float4
// column over the partition's items (in item order), eight loads in flight.
__global__ void commit_slice_kernel(CommitArgs a, int64_t slice4) {
  grid_dep_launch();
  grid_dep_wait();
  const int e = blockIdx.y;
  const int i0 = a.e_item0[e], i1 = a.e_item0[e + 1];
  const int64_t P4 = a.P / 4;
  const int64_t c0 = (int64_t)blockIdx.x * slice4;
  if (c0 >= P4) return;
  const int64_t w4 = c0 + slice4 <= P4 ? slice4 : P4 - c0;
  const float4* src = reinterpret_cast<const float4*>(a.partials);
  const float sc = a.e_scale[e];
  const int32_t* dest = a.e_dest + (int64_t)e * a.ndest;
  for (int64_t j = threadIdx.x; j < w4; j += blockDim.x) {
    const int64_t p = c0 + j;
    float4 acc = f4zero();
    for (int it = i0; it < i1; it += 8) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = it + u < i1 ? __ldcg(src + (int64_t)(it + u) * P4 + p) : f4zero();
#pragma unroll
      for (int u = 0; u < 8; ++u) acc = f4add(acc, v[u]);
    }
    acc = make_float4(acc.x * sc, acc.y * sc, acc.z * sc, acc.w * sc);
    for (int k = 0; k < a.ndest; ++k) {
      const int dst = dest[k];
      if (dst >= 0) reinterpret_cast<float4*>(a.store)[(int64_t)dst * P4 + p] = acc;
    }
  }
}

template <typename K, typename... Args>
static cudaError_t launch_maybe_pdl(bool pdl, K kern, dim3 grid, dim3 block, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

cudaError_t launch_commit(const CommitArgs& a, cudaStream_t st, bool pdl) {
  if (a.nE <= 0) return cudaSuccess;
  const int64_t P4 = a.P / 4;
  const int threads = 128;
  // one float4 column per thread: slices of 128 columns per CTA, one grid row
  // per partition (the sums are short and latency-bound: many CTAs)
  const int64_t slice4 = threads;
  const int64_t bx = (P4 + slice4 - 1) / slice4;
  return launch_maybe_pdl(pdl, commit_slice_kernel, dim3((unsigned)bx, (unsigned)a.nE), dim3(threads), st, a, slice4);
}

__global__ void __launch_bounds__(kDecX * kDecY) decode_kernel(DecodeArgs a) {
  __shared__ DecodePlan pl;
  __shared__ float4 red[kDecY][kDecX];
  grid_dep_launch();
  if (threadIdx.x < 32) derive_plan_warp(a, pl, threadIdx.x);   // needs only the mask
  __syncthreads();
  grid_dep_wait();
  if (blockIdx.x == 0 && threadIdx.x < 32) write_coeffs_warp(a, threadIdx.x);
  auto bar = [] { __syncthreads(); };
  decode_chunks(a, pl, red, (int)threadIdx.x, blockIdx.x, gridDim.x, bar);
}

// Sum of cnt float4 loads base[off(j)], j = 0..cnt-1, issued eight at a time
// so that each thread keeps eight independent loads in flight.
template <class Off>
__device__ __forceinline__ float4 sum_loads8(const float4* base, int cnt, Off off) {
  float4 acc = f4zero();
  for (int j0 = 0; j0 < cnt; j0 += 8) {
    float4 v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = j0 + j < cnt ? __ldcg(base + off(j0 + j)) : f4zero();
#pragma unroll
    for (int j = 0; j < 8; ++j) acc = f4add(acc, v[j]);
  }
  return acc;
}

// Decode + SGD for large P: one thread per float4 column, grid-stride, no
// barriers after the plan.  Same arithmetic as decode_chunks.
__global__ void __launch_bounds__(256) decode_wide_kernel(DecodeArgs a) {
  __shared__ DecodePlan pl;
  grid_dep_launch();
  if (threadIdx.x < 32) derive_plan_warp(a, pl, threadIdx.x);   // needs only the mask
  __syncthreads();
  grid_dep_wait();
  if (blockIdx.x == 0 && threadIdx.x < 32) write_coeffs_warp(a, threadIdx.x);
  const int64_t P4 = a.P / 4;
  const int c = a.c;
  const float4* store = reinterpret_cast<const float4*>(a.store);
  float4* U = reinterpret_cast<float4*>(a.U);
  const int64_t slotP = (int64_t)c * P4;           // float4s per store
  if (a.pre && a.u_ready && a.slot >= 0) {
    // the slots other than o_t were summed early: add U[o_t] and the
    // deviating stores' slot o_t
    const float4* pre = reinterpret_cast<const float4*>(a.pre);
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P4; p += (int64_t)gridDim.x * blockDim.x) {
      float4 g = f4fma(pl.B, __ldcg(U + (int64_t)a.slot * P4 + p), __ldcg(pre + p));
      const float4* cur = store + (int64_t)a.slot * P4 + p;
      for (int q0 = 0; q0 < pl.ndev; q0 += 8) {
        float4 v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = q0 + j < pl.ndev ? __ldcg(cur + (int64_t)pl.dev[q0 + j] * slotP) : f4zero();
#pragma unroll
        for (int j = 0; j < 8; ++j)
          if (q0 + j < pl.ndev) g = f4fma(pl.devc[q0 + j], v[j], g);
      }
      float4 w = __ldcg(reinterpret_cast<const float4*>(a.w) + p);
      w = f4fma(-a.lr, g, w);
      store_outputs(a, p, g, w);
    }
    return;
  }
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P4; p += (int64_t)gridDim.x * blockDim.x) {
    float4 V = f4zero();
    if (a.slot < 0) {
      for (int o = 0; o < c; ++o) {
        const float4 u = sum_loads8(store + (int64_t)o * P4 + p, a.owners, [&](int r) { return (int64_t)r * slotP; });
        U[(int64_t)o * P4 + p] = u;
        V = f4add(V, u);
      }
    } else {
      const int skip = a.u_ready ? -1 : a.slot;      // the slot re-summed below
      const int nu = a.u_ready ? c : c - 1;
      V = sum_loads8(U + p, nu, [&](int j) { return (int64_t)(skip >= 0 && j >= skip ? j + 1 : j) * P4; });
      if (!a.u_ready) {
        const float4 u =
            sum_loads8(store + (int64_t)a.slot * P4 + p, a.owners, [&](int r) { return (int64_t)r * slotP; });
        U[(int64_t)a.slot * P4 + p] = u;
        V = f4add(V, u);
      }
    }
    float4 D = f4zero();
    for (int q = 0; q < pl.ndev; ++q) {
      const float4 Cr = sum_loads8(store + (int64_t)pl.dev[q] * slotP + p, c, [&](int o) { return (int64_t)o * P4; });
      D = f4fma(pl.devc[q], Cr, D);
    }
    const float4 g = f4fma(pl.B, V, D);
    float4 w = __ldcg(reinterpret_cast<const float4*>(a.w) + p);
    w = f4fma(-a.lr, g, w);
    store_outputs(a, p, g, w);
  }
}

// Columns from which the one-thread-per-column decode is used.
constexpr int64_t kWideDecodeMinP4 = 1 << 18;

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st, bool pdl, int sm_count) {
  if (a.n > kMaxWorkers || a.owners > kMaxWorkers) return cudaErrorInvalidValue;
  if (a.P / 4 >= kWideDecodeMinP4) {
    int64_t blocks = (a.P / 4 + 255) / 256;
    if (blocks > (int64_t)sm_count * 8) blocks = (int64_t)sm_count * 8;
    return launch_maybe_pdl(pdl, decode_wide_kernel, dim3((unsigned)blocks), dim3(256), st, a);
  }
  const int64_t P4 = a.P / 4;
  int64_t chunks = (P4 + kDecX - 1) / kDecX;
  int64_t blocks = chunks < (int64_t)sm_count * 8 ? chunks : (int64_t)sm_count * 8;
  if (blocks < 1) blocks = 1;
  return launch_maybe_pdl(pdl, decode_kernel, dim3((unsigned)blocks), dim3(kDecX * kDecY), st, a);
}

// ---------------------------------------------------------------------------
// fp32 -> bf16 (round to nearest even)
// ---------------------------------------------------------------------------
__global__ void f32_to_bf16_kernel(const float* __restrict__ src, uint16_t* __restrict__ dst, int64_t count) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count; i += (int64_t)gridDim.x * blockDim.x) {
    __nv_bfloat16 b = __float2bfloat16_rn(src[i]);
    dst[i] = *reinterpret_cast<uint16_t*>(&b);
  }
}

cudaError_t launch_f32_to_bf16(const float* src, uint16_t* dst, int64_t count, cudaStream_t st) {
  if (count <= 0) return cudaSuccess;
  int64_t blocks = (count + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  f32_to_bf16_kernel<<<(unsigned)blocks, 256, 0, st>>>(src, dst, count);
  return cudaGetLastError();
}

}  // namespace pgc
