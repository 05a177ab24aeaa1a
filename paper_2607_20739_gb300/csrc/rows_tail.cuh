// The fused tail of the whole-row few-class softmax kernel (softmax_rows.cu):
// after the grid's gradient partials are written, the same grid commits them
// into the stores and decodes (§IV-A, §V-B), fused with the SGD update
// (§III).  Every CTA takes a slice of the float4 columns; the grid must be
// co-resident (one CTA per SM) for its barrier.
#pragma once

#include "tail.cuh"

namespace pgc {

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// Every CTA of the (co-resident) grid arrives on *ctr and waits until all
// have; bounded.  Called by all threads of the CTA.
static __device__ bool grid_barrier(int* ctr, int* status, int* flag) {
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    atomic_add_acq_rel(ctr, 1);
    const int target = (int)gridDim.x;
    if (ld_acquire(ctr) < target) {
      const uint64_t t0 = globaltimer_ns();
      for (uint32_t it = 0;; ++it) {
        if (ld_acquire(ctr) >= target) break;
        if (it > kWaitMaxIters || ((it & 63u) == 63u && globaltimer_ns() - t0 > kWaitMaxNs)) {
          atomicOr(status, kErrWaitTimeout);
          ok = 0;
          break;
        }
      }
    }
    *flag = ok;
  }
  __syncthreads();
  return *flag != 0;
}

constexpr int kTailMaxC = 4;   // slots per store on the fused tail's short route

// Commit, then decode + SGD, for this CTA's slice of the columns.  Called by
// all threads of the CTA after its partials are written.  plan: shared
// memory for the decode plan; gs_area / gs_bytes: idle shared memory for
// the committed gradients of the short route; bar_flag: a shared int.
__device__ __forceinline__ void rows_fused_tail(const RowsArgs& a, DecodePlan& plan, uint8_t* gs_area,
                                                int64_t gs_bytes, int* bar_flag) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // ---- fused tail: commit, then decode + SGD --------------------------------
  // After one grid barrier (every partial written) each CTA commits every
  // evaluated partition for its own slice of the float4 columns and then
  // decodes that slice: a column's decode reads only that column of the
  // stores and slot totals, all written by this CTA, so a CTA barrier
  // stands in for a second grid barrier.
  //
  // Steady steps (one store per evaluated partition, every store's slot o_t
  // refreshed) take a shorter route: the slot totals this step leaves as
  // they are, and beta, are loaded before the grid barrier, and the
  // committed gradients reach the decode through shared memory (the slots'
  // area, idle after the tiles), so U[o_t] = sum_e g_e needs no second
  // round trip through L2.
  if (warp == 0) derive_plan_warp(a.dec, plan, lane);   // needs only the mask
  const int64_t P4 = a.P / 4;
  const int64_t q0 = P4 * blockIdx.x / gridDim.x, q1 = P4 * (blockIdx.x + 1) / gridDim.x, nq = q1 - q0;
  const DecodeArgs& dc = a.dec;
  const bool fast = dc.slot >= 0 && !dc.u_ready && a.ndest == 1 && a.nE == dc.owners && dc.c <= kTailMaxC &&
                    nq <= (int64_t)blockDim.x && (int64_t)a.nE * nq * 16 <= gs_bytes;
  float4* gs = reinterpret_cast<float4*>(gs_area);           // [nE][nq] committed gradients (fast route)
  float4 up[kTailMaxC], wv = f4zero();
  const int64_t pq = q0 + threadIdx.x;
  if (fast && (int64_t)threadIdx.x < nq) {
    const float4* U4 = reinterpret_cast<const float4*>(dc.U);
#pragma unroll
    for (int o = 0; o < kTailMaxC; ++o) up[o] = (o < dc.c && o != dc.slot) ? __ldcg(U4 + (int64_t)o * P4 + pq) : f4zero();
    wv = __ldcg(reinterpret_cast<const float4*>(dc.w) + pq);
  }
  bool ok = grid_barrier(a.counters, a.status, bar_flag);   // every partial is written
  if (ok) {
    const float4* src = reinterpret_cast<const float4*>(a.partials);
    for (int64_t x = threadIdx.x; x < (int64_t)a.nE * nq; x += blockDim.x) {
      const int e = (int)(x / nq);
      const int64_t p = q0 + (x - (int64_t)e * nq);
      const int i0 = a.e_item0[e], i1 = a.e_item0[e + 1];
      float4 acc = f4zero();
      // a partition has about (pairs / partitions) + 1 items: one batch of
      // loads in flight covers it
      for (int it = i0; it < i1; it += 16) {
        float4 v[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = it + u < i1 ? __ldcg(src + (int64_t)(it + u) * P4 + p) : f4zero();
#pragma unroll
        for (int u = 0; u < 16; ++u) acc = f4add(acc, v[u]);
      }
      const float sc = a.e_scale[e];
      acc = make_float4(acc.x * sc, acc.y * sc, acc.z * sc, acc.w * sc);
      for (int k = 0; k < a.ndest; ++k) {
        const int dst = a.e_dest[(int64_t)e * a.ndest + k];
        if (dst >= 0) reinterpret_cast<float4*>(a.store)[(int64_t)dst * P4 + p] = acc;
      }
      if (fast) gs[x] = acc;
    }
    __syncthreads();                   // this CTA's stores (and gs) are visible to all its threads
    if (blockIdx.x == 0 && warp == 0) write_coeffs_warp(a.dec, lane);
    if (!fast) {
      decode_columns(a.dec, plan, q0, q1, (int)threadIdx.x, (int)blockDim.x);
    } else if ((int64_t)threadIdx.x < nq) {
      // U[o_t] = sum over the evaluated partitions of their new gradients
      float4 un = f4zero();
      for (int e = 0; e < a.nE; ++e) un = f4add(un, gs[(int64_t)e * nq + threadIdx.x]);
      reinterpret_cast<float4*>(dc.U)[(int64_t)dc.slot * P4 + pq] = un;
      float4 V = f4zero(), D = f4zero();
#pragma unroll
      for (int o = 0; o < kTailMaxC; ++o)
        if (o < dc.c) V = f4add(V, o == dc.slot ? un : up[o]);
      const float4* st4 = reinterpret_cast<const float4*>(dc.store);
      for (int q = 0; q < plan.ndev; ++q) {
        float4 Cr = f4zero();
        for (int o = 0; o < dc.c; ++o) Cr = f4add(Cr, __ldcg(st4 + ((int64_t)plan.dev[q] * dc.c + o) * P4 + pq));
        D = f4fma(plan.devc[q], Cr, D);
      }
      const float4 g = f4fma(plan.B, V, D);
      store_outputs(dc, pq, g, f4fma(-dc.lr, g, wv));
    }
    __syncthreads();
    // the last CTA out resets the counters for the next step
    if (threadIdx.x == 0 && atomic_add_acq_rel(a.counters + 2, 1) == (int)gridDim.x - 1) {
      a.counters[0] = 0;
      a.counters[2] = 0;
      __threadfence();
    }
  }
}

}  // namespace pgc
