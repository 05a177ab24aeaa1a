// K4 — store commit: g_e = (1/m_e) * sum of the work items' partial sums,
//      written into the gradient store of every worker (or FR group) that
//      keeps this copy (§VI-A: each worker keeps its latest gradient per
//      partition).
// K5+K6 — decode: the coefficients of the received coded gradients are
//      derived on the device from the straggler mask (§IV-A: one coded
//      gradient per FR group, times 1/n; §V-B: every received CR coded
//      gradient times 1/((n-s)c)), the aggregate is formed, and the SGD
//      update beta <- beta - eta * ghat (§III) is applied in the same pass.
//
// Decode arithmetic.  Coded gradient of store r: C_r = sum_o store[r][o]
// (all coefficients 1, §IV-A / §V-B).  Slot totals U[o] = sum_r store[r][o].
// With b_r the summed coefficient of the workers sharing store r and a
// baseline B,
//     ghat = sum_r b_r C_r = B * sum_o U[o] + sum_{r: b_r != B} (b_r - B) C_r.
// FR: every group's coefficient is 1/n = B, so ghat = (1/n) sum_o U[o].
// CR: B = 1/((n-s)c) and only the s stragglers deviate (b_r = 0).
// This reads (c + s*c) gradients instead of the (n - s) * c of the literal
// sum; U[o_t] is refreshed from the stores just written.
#include "dev_common.cuh"
#include "pgc_internal.h"
#include "../../include/pgc.h"

namespace pgc {

__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 f4fma(float s, float4 a, float4 b) {
  return make_float4(fmaf(s, a.x, b.x), fmaf(s, a.y, b.y), fmaf(s, a.z, b.z), fmaf(s, a.w, b.w));
}

// ---------------------------------------------------------------------------
// K4 commit
// ---------------------------------------------------------------------------
__global__ void commit_kernel(CommitArgs a) {
  const int e = blockIdx.y;
  const int64_t P4 = a.P / 4;
  const int i0 = a.e_item0[e], i1 = a.e_item0[e + 1];
  const float sc = a.e_scale[e];
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P4; p += (int64_t)gridDim.x * blockDim.x) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    const float4* src = reinterpret_cast<const float4*>(a.partials) + p;
    int it = i0;
    for (; it + 4 <= i1; it += 4) {
      const float4 v0 = src[(int64_t)(it + 0) * P4];
      const float4 v1 = src[(int64_t)(it + 1) * P4];
      const float4 v2 = src[(int64_t)(it + 2) * P4];
      const float4 v3 = src[(int64_t)(it + 3) * P4];
      acc = f4add(f4add(f4add(f4add(acc, v0), v1), v2), v3);
    }
    for (; it < i1; ++it) acc = f4add(acc, src[(int64_t)it * P4]);
    acc = make_float4(acc.x * sc, acc.y * sc, acc.z * sc, acc.w * sc);
    for (int j = 0; j < a.ndest; ++j) {
      const int dst = a.e_dest[e * a.ndest + j];
      if (dst >= 0) reinterpret_cast<float4*>(a.store)[(int64_t)dst * P4 + p] = acc;
    }
  }
}

cudaError_t launch_commit(const CommitArgs& a, cudaStream_t st) {
  if (a.nE <= 0) return cudaSuccess;
  const int64_t P4 = a.P / 4;
  const int threads = 128;
  int64_t bx = (P4 + threads - 1) / threads;
  if (bx > 4096) bx = 4096;
  commit_kernel<<<dim3((unsigned)bx, (unsigned)a.nE), threads, 0, st>>>(a);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// K5+K6 decode + SGD
// ---------------------------------------------------------------------------
constexpr int kDecThreads = 256;

struct DecodeShared {
  float a[kMaxWorkers];        // per-worker coefficient a_i
  float b[kMaxWorkers];        // per-store summed coefficient b_r
  int dev[kMaxWorkers];        // stores whose b_r != B, ascending
  float devc[kMaxWorkers];     // b_r - B for those stores
  int ndev;
  float B;
};

__device__ __forceinline__ bool straggles(const MaskBits& m, int i) { return (m.w[i >> 5] >> (i & 31)) & 1u; }

// Derive a_i, b_r, B and the deviating stores from the mask (§IV-A, §V-B).
__device__ void derive_coefficients(const DecodeArgs& a, DecodeShared& sh) {
  const int tid = threadIdx.x;
  const int c = a.c;
  if (a.scheme == PGC_CR) {
    const float A = 1.0f / (float)((a.n - a.s) * c);     // 1/(n mu), mu = (n-s)c/n
    for (int i = tid; i < a.n; i += blockDim.x) {
      const float ai = straggles(a.mask, i) ? 0.f : A;
      sh.a[i] = ai;
      sh.b[i] = ai;                                        // one store per worker
    }
    if (tid == 0) sh.B = A;
  } else {
    const float inv_n = 1.0f / (float)a.n;
    // representative of group g: lowest-index worker of the group that is
    // not a straggler; the group's coefficient is 1/n
    for (int g = tid; g < a.owners; g += blockDim.x) {
      int rep = -1;
      for (int l = 0; l < c && rep < 0; ++l)
        if (!straggles(a.mask, g * c + l)) rep = g * c + l;
      float bg = 0.f;
      for (int l = 0; l < c; ++l) {
        const float ai = (g * c + l == rep) ? inv_n : 0.f;
        sh.a[g * c + l] = ai;
        bg += ai;
      }
      sh.b[g] = bg;
      if (rep < 0) atomicOr(a.status, kErrBadMask);
    }
    if (tid == 0) sh.B = inv_n;
  }
  __syncthreads();
  // stragglers counted by every CTA; a wrong count flags the status word
  if (tid < 32) {
    int cnt = 0;
    for (int i = tid; i < a.n; i += 32) cnt += straggles(a.mask, i) ? 1 : 0;
    for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    // deviating stores, in ascending order, by warp ballots
    int nd = 0;
    for (int base = 0; base < a.owners; base += 32) {
      const int r = base + tid;
      const bool devr = r < a.owners && sh.b[r] != sh.B;
      const unsigned bal = __ballot_sync(0xffffffffu, devr);
      if (devr) {
        const int pos = nd + __popc(bal & ((1u << tid) - 1u));
        sh.dev[pos] = r;
        sh.devc[pos] = sh.b[r] - sh.B;
      }
      nd += __popc(bal);
    }
    if (tid == 0) {
      sh.ndev = nd;
      if (cnt != a.s) atomicOr(a.status, kErrBadMask);
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(kDecThreads) decode_kernel(DecodeArgs a) {
  __shared__ DecodeShared sh;
  derive_coefficients(a, sh);
  if (blockIdx.x == 0 && a.coeff_out)
    for (int i = threadIdx.x; i < a.n; i += blockDim.x) a.coeff_out[i] = sh.a[i];

  const int64_t P4 = a.P / 4;
  const int c = a.c;
  const float B = sh.B;
  const int ndev = sh.ndev;
  const float4* store = reinterpret_cast<const float4*>(a.store);
  float4* U = reinterpret_cast<float4*>(a.U);
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P4; p += (int64_t)gridDim.x * blockDim.x) {
    float4 V = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int o = 0; o < c; ++o) {
      float4 u;
      if (a.slot < 0 || o == a.slot) {
        u = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int r = 0; r < a.owners; ++r) u = f4add(u, store[((int64_t)r * c + o) * P4 + p]);
        U[(int64_t)o * P4 + p] = u;
      } else {
        u = U[(int64_t)o * P4 + p];
      }
      V = f4add(V, u);
    }
    float4 g = make_float4(B * V.x, B * V.y, B * V.z, B * V.w);
    for (int q = 0; q < ndev; ++q) {
      const int r = sh.dev[q];
      float4 C = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int o = 0; o < c; ++o) C = f4add(C, store[((int64_t)r * c + o) * P4 + p]);
      g = f4fma(sh.devc[q], C, g);
    }
    float4 w = reinterpret_cast<float4*>(a.w)[p];
    w = f4fma(-a.lr, g, w);
    reinterpret_cast<float4*>(a.w)[p] = w;
    reinterpret_cast<float4*>(a.gout)[p] = g;
    if (a.wb) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(w.x, w.y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(w.z, w.w);
      uint2 pk;
      pk.x = *reinterpret_cast<uint32_t*>(&lo);
      pk.y = *reinterpret_cast<uint32_t*>(&hi);
      reinterpret_cast<uint2*>(a.wb)[p] = pk;
    }
  }
}

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  if (a.n > kMaxWorkers || a.owners > kMaxWorkers) return cudaErrorInvalidValue;
  const int64_t P4 = a.P / 4;
  int64_t blocks = (P4 + kDecThreads - 1) / kDecThreads;
  if (blocks > 1216) blocks = 1216;
  if (blocks < 1) blocks = 1;
  decode_kernel<<<(unsigned)blocks, kDecThreads, 0, st>>>(a);
  return cudaGetLastError();
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
