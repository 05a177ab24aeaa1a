// Block-level pieces of a step's tail, shared by the standalone commit /
// decode kernels and by the gradient kernel's fused tail:
//
//   commit_block      g_e = scale * (ordered sum of partition e's partial
//                     sums), written to each store that keeps this copy
//                     (§VI-A: every worker keeps its latest gradients).
//   derive_plan_warp  the decode coefficients from the straggler mask, by one
//                     warp (§IV-A FR: one coded gradient per group, times
//                     1/n; §V-B CR: every received coded gradient, times
//                     1/(n mu) = 1/((n-s)c)).
//   decode_columns /  ghat = B * sum_o U[o] + sum_{stores r with b_r != B}
//   decode_chunks     (b_r - B) * sum_o store[r][o], fused with the SGD update
//                     beta <- beta - eta * ghat (§III); U[o_t] is refreshed.
//
// Decode arithmetic.  Coded gradient of store r: C_r = sum_o store[r][o]
// (every coefficient 1, §IV-A / §V-B).  Slot totals U[o] = sum_r store[r][o].
// With b_r the summed coefficient of the workers sharing store r and a
// baseline B,  ghat = sum_r b_r C_r = B sum_o U[o] + sum_{b_r != B} (b_r - B) C_r.
// FR: every group's coefficient is 1/n = B, so ghat = (1/n) sum_o U[o].
// CR: B = 1/((n-s)c) and only the s stragglers deviate (b_r = 0).  This reads
// (owners + c + s c) gradients instead of the (n - s) c of the literal sum.
//
// Data written by other CTAs of the same grid is read with ld.global.cg (L2)
// after a release (writer fence + atomic) / acquire (reader atomic + fence)
// handshake.
#pragma once

#include "dev_common.cuh"
#include "pgc_internal.h"
#include "pgc.h"

namespace pgc {

__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 f4fma(float s, float4 a, float4 b) {
  return make_float4(fmaf(s, a.x, b.x), fmaf(s, a.y, b.y), fmaf(s, a.z, b.z), fmaf(s, a.w, b.w));
}
__device__ __forceinline__ float4 f4zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }

__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------------------
// commit
// ---------------------------------------------------------------------------
__device__ __forceinline__ void commit_block(const float* partials, int64_t P, int i0, int i1, float scale,
                                             const int32_t* dest, int ndest, float* store, int tid, int nthr) {
  constexpr int kB = 20;          // partials loaded per batch (one item per SM: 152 / 8 = 19 at n = 8)
  const int64_t P4 = P / 4;
  const float4* src = reinterpret_cast<const float4*>(partials);
  for (int64_t p = tid; p < P4; p += nthr) {
    float4 acc = f4zero();
    for (int it = i0; it < i1; it += kB) {
      float4 v[kB];
#pragma unroll
      for (int j = 0; j < kB; ++j) v[j] = it + j < i1 ? __ldcg(src + (int64_t)(it + j) * P4 + p) : f4zero();
#pragma unroll
      for (int j = 0; j < kB; ++j) acc = f4add(acc, v[j]);
    }
    acc = make_float4(acc.x * scale, acc.y * scale, acc.z * scale, acc.w * scale);
    for (int j = 0; j < ndest; ++j) {
      const int dst = dest[j];
      if (dst >= 0) reinterpret_cast<float4*>(store)[(int64_t)dst * P4 + p] = acc;
    }
  }
}

// ---------------------------------------------------------------------------
// decode plan
// ---------------------------------------------------------------------------
struct DecodePlan {
  float B;                     // baseline coefficient
  int ndev;                    // stores whose summed coefficient differs from B
  int dev[kMaxWorkers];        // ascending
  float devc[kMaxWorkers];     // b_r - B
};

__device__ __forceinline__ bool straggles(const MaskBits& m, int i) { return (m.w[i >> 5] >> (i & 31)) & 1u; }

// FR: representative of group g = lowest-index non-straggler, or -1.
__device__ __forceinline__ int fr_rep(const DecodeArgs& a, int g) {
  for (int l = 0; l < a.c; ++l)
    if (!straggles(a.mask, g * a.c + l)) return g * a.c + l;
  return -1;
}

// One warp derives the plan; invalid masks set kErrBadMask.  It depends only
// on the mask, so it can run before the step's gradients exist.  Plan: a
// DecodePlan, or a struct of the same members with shorter dev / devc arrays
// (more deviating stores than they hold also set kErrBadMask).
template <class Plan>
__device__ __forceinline__ void derive_plan_warp(const DecodeArgs& a, Plan& pl, int lane) {
  constexpr int kCap = (int)(sizeof(pl.dev) / sizeof(pl.dev[0]));
  const bool cr = a.scheme == PGC_CR;
  const float A = cr ? 1.0f / (float)((a.n - a.s) * a.c) : 1.0f / (float)a.n;
  int cnt = 0;
  for (int i = lane; i < a.n; i += 32) cnt += straggles(a.mask, i) ? 1 : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  int nd = 0;
  for (int base = 0; base < a.owners; base += 32) {
    const int r = base + lane;
    float br = A;
    if (r < a.owners) {
      if (cr) {
        br = straggles(a.mask, r) ? 0.f : A;         // one store per worker
      } else {
        const bool alive = fr_rep(a, r) >= 0;        // 1/n from the group's representative
        br = alive ? A : 0.f;
        if (!alive) atomicOr(a.status, kErrBadMask);
      }
    }
    const bool devr = r < a.owners && br != A;
    const unsigned bal = __ballot_sync(0xffffffffu, devr);
    if (devr) {
      const int pos = nd + __popc(bal & ((1u << lane) - 1u));
      if (pos < kCap) {
        pl.dev[pos] = r;
        pl.devc[pos] = br - A;
      }
    }
    nd += __popc(bal);
  }
  if (lane == 0) {
    pl.ndev = nd < kCap ? nd : kCap;
    pl.B = A;
    if (cnt != a.s || nd > kCap) atomicOr(a.status, kErrBadMask);
  }
  __syncwarp();
}

// The per-worker coefficients a_i, written by one warp of the decoding CTA.
__device__ __forceinline__ void write_coeffs_warp(const DecodeArgs& a, int lane) {
  if (!a.coeff_out) return;
  const bool cr = a.scheme == PGC_CR;
  const float A = cr ? 1.0f / (float)((a.n - a.s) * a.c) : 1.0f / (float)a.n;
  for (int i = lane; i < a.n; i += 32)
    a.coeff_out[i] = cr ? (straggles(a.mask, i) ? 0.f : A) : (fr_rep(a, i / a.c) == i ? A : 0.f);
}

__device__ __forceinline__ void store_outputs(const DecodeArgs& a, int64_t p, float4 g, float4 w) {
  reinterpret_cast<float4*>(a.w)[p] = w;
  reinterpret_cast<float4*>(a.gout)[p] = g;
  if (a.w_user) reinterpret_cast<float4*>(a.w_user)[p] = w;
  if (a.g_user) reinterpret_cast<float4*>(a.g_user)[p] = g;
  if (a.wb) {
    __nv_bfloat162 lo = __floats2bfloat162_rn(w.x, w.y);
    __nv_bfloat162 hi = __floats2bfloat162_rn(w.z, w.w);
    uint2 pk;
    pk.x = *reinterpret_cast<uint32_t*>(&lo);
    pk.y = *reinterpret_cast<uint32_t*>(&hi);
    reinterpret_cast<uint2*>(a.wb)[p] = pk;
  }
}

// Decode + SGD of the float4 columns [q0, q1), every column handled by one
// thread (tid of nthr) and no barriers.  When the counts fit the unrolled
// bounds all loads of a column are issued back to back; otherwise plain loops.
__device__ __forceinline__ void decode_columns(const DecodeArgs& a, const DecodePlan& pl, int64_t q0, int64_t q1,
                                               int tid, int nthr) {
  constexpr int kMaxO = 8, kMaxC = 4, kMaxD = 4;
  const int64_t P4 = a.P / 4;
  const int c = a.c;
  const float B = pl.B;
  const int ndev = pl.ndev;
  const float4* store = reinterpret_cast<const float4*>(a.store);
  float4* U = reinterpret_cast<float4*>(a.U);
  const bool small = a.owners <= kMaxO && c <= kMaxC && ndev <= kMaxD && a.slot >= 0 && !a.u_ready;
  for (int64_t p = q0 + tid; p < q1; p += nthr) {
    float4 V = f4zero(), D = f4zero();
    if (small) {
      float4 u[kMaxO], o4[kMaxC], dv[kMaxD][kMaxC];
#pragma unroll
      for (int r = 0; r < kMaxO; ++r)
        u[r] = r < a.owners ? __ldcg(store + ((int64_t)r * c + a.slot) * P4 + p) : f4zero();
#pragma unroll
      for (int o = 0; o < kMaxC; ++o)
        o4[o] = (o < c && o != a.slot) ? __ldcg(U + (int64_t)o * P4 + p) : f4zero();
#pragma unroll
      for (int q = 0; q < kMaxD; ++q)
#pragma unroll
        for (int o = 0; o < kMaxC; ++o)
          dv[q][o] = (q < ndev && o < c) ? __ldcg(store + ((int64_t)pl.dev[q] * c + o) * P4 + p) : f4zero();
      float4 un = f4zero();
#pragma unroll
      for (int r = 0; r < kMaxO; ++r) un = f4add(un, u[r]);
      U[(int64_t)a.slot * P4 + p] = un;
#pragma unroll
      for (int o = 0; o < kMaxC; ++o) V = f4add(V, o < c && o == a.slot ? un : o4[o]);
#pragma unroll
      for (int q = 0; q < kMaxD; ++q) {
        float4 Cr = f4zero();
#pragma unroll
        for (int o = 0; o < kMaxC; ++o) Cr = f4add(Cr, dv[q][o]);
        if (q < ndev) D = f4fma(pl.devc[q], Cr, D);
      }
    } else {
      for (int o = 0; o < c; ++o) {
        if (a.slot < 0 || (o == a.slot && !a.u_ready)) {
          float4 u = f4zero();
          for (int r = 0; r < a.owners; ++r) u = f4add(u, __ldcg(store + ((int64_t)r * c + o) * P4 + p));
          U[(int64_t)o * P4 + p] = u;
          V = f4add(V, u);
        } else {
          V = f4add(V, __ldcg(U + (int64_t)o * P4 + p));
        }
      }
      for (int q = 0; q < ndev; ++q) {
        float4 Cr = f4zero();
        for (int o = 0; o < c; ++o) Cr = f4add(Cr, __ldcg(store + ((int64_t)pl.dev[q] * c + o) * P4 + p));
        D = f4fma(pl.devc[q], Cr, D);
      }
    }
    const float4 g = f4fma(B, V, D);
    float4 w = __ldcg(reinterpret_cast<const float4*>(a.w) + p);
    w = f4fma(-a.lr, g, w);
    store_outputs(a, p, g, w);
  }
}

// Decode + SGD over chunks q0, q0 + qstride, ... of kDecX float4 columns, the
// stores split over kDecY thread rows (for large P, many CTAs).  Must be
// called by exactly kDecX * kDecY threads, all of which pass every bar().
constexpr int kDecX = 32;
constexpr int kDecY = 8;

template <class Bar>
__device__ void decode_chunks(const DecodeArgs& a, const DecodePlan& pl, float4 (*red)[kDecX], int tid, int64_t q0,
                              int64_t qstride, Bar bar) {
  const int x = tid % kDecX, y = tid / kDecX;
  const int64_t P4 = a.P / 4;
  const int64_t nq = (P4 + kDecX - 1) / kDecX;
  const int c = a.c;
  const float B = pl.B;
  const int ndev = pl.ndev;
  const float4* store = reinterpret_cast<const float4*>(a.store);
  float4* U = reinterpret_cast<float4*>(a.U);
  for (int64_t q = q0; q < nq; q += qstride) {
    const int64_t p = q * kDecX + x;
    const bool inb = p < P4;
    float4 V = f4zero();
    for (int o = 0; o < c; ++o) {
      if (a.slot < 0 || (o == a.slot && !a.u_ready)) {
        float4 part = f4zero();
        if (inb)
          for (int r = y; r < a.owners; r += kDecY) part = f4add(part, __ldcg(store + ((int64_t)r * c + o) * P4 + p));
        red[y][x] = part;
        bar();
        if (y == 0) {
          float4 u = red[0][x];
#pragma unroll
          for (int j = 1; j < kDecY; ++j) u = f4add(u, red[j][x]);
          if (inb) U[(int64_t)o * P4 + p] = u;
          V = f4add(V, u);
        }
        bar();
      } else if (y == 0 && inb) {
        V = f4add(V, __ldcg(U + (int64_t)o * P4 + p));
      }
    }
    float4 dv = f4zero();
    if (inb)
      for (int qq = y; qq < ndev; qq += kDecY) {
        const int r = pl.dev[qq];
        float4 Cr = f4zero();
        for (int o = 0; o < c; ++o) Cr = f4add(Cr, __ldcg(store + ((int64_t)r * c + o) * P4 + p));
        dv = f4fma(pl.devc[qq], Cr, dv);
      }
    red[y][x] = dv;
    bar();
    if (y == 0 && inb) {
      float4 D = red[0][x];
#pragma unroll
      for (int j = 1; j < kDecY; ++j) D = f4add(D, red[j][x]);
      const float4 g = f4fma(B, V, D);
      float4 w = __ldcg(reinterpret_cast<const float4*>(a.w) + p);
      w = f4fma(-a.lr, g, w);
      store_outputs(a, p, g, w);
    }
    bar();
  }
}

}  // namespace pgc
