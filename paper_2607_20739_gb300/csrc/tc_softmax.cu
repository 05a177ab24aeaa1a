// Logits GEMM with the softmax residual in its epilogue (§III with f = log
// sum_k exp(w_k.x) - w_y.x): for every 128-row tile of the evaluated
// partitions, R = softmax(X Wb^T) - onehot(y) in bf16, written straight to
// the R buffer that the gradient contraction reads; the logits never leave
// the chip.
//
// A cluster of NT CTAs (NT = padded classes / 256, one 256-class N tile each)
// computes one row tile at a time.  The X tile is common to the cluster: each
// CTA loads 128/NT of its rows and multicasts them to all NT CTAs, and loads
// its own 256 x 64 W tile, into a 4-stage ring (2-D TMA, 128-byte swizzle);
// a stage is refilled once all NT CTAs' MMAs have read it.  Warp 1 issues
// tcgen05.mma (M = 128 rows, N = 256 classes, K = 16) into one of two TMEM
// accumulators.  Warps 2-5 (one row per thread) drain the other:
//   pass 1  the row's maximum m and sum of exp(z - m) over this CTA's classes;
//   the NT partial (m, s) pairs of every row are sent to all CTAs of the
//   cluster with st.async into distributed shared memory (two buffers; a
//   buffer is rewritten only after every CTA's epilogue has read it);
//   pass 2  r = exp(z - M) / S - [class == y] with the row's combined M, S,
//   rounded to bf16, staged as 32 x 64 boxes in swizzled shared memory and
//   written with TMA stores.  Rows past the partition and classes past K
//   inside a box are written as zeros (the gradient contraction reads whole
//   64-row blocks); boxes wholly past K are not written (the buffer starts
//   zeroed).  The grid also zeroes the slot total that the gradient
//   contraction accumulates into.
// Every wait is bounded; the cluster barrier at the end keeps every CTA alive
// until no peer can still write into it.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "tc_common.cuh"

namespace pgc {

namespace {

constexpr int kFM = 128, kFN = 256, kFK = 64;
constexpr int kFStages = 4;
constexpr uint32_t kFA = kFM * kFK * 2;        // 16 KB A tile per stage
constexpr uint32_t kFB = kFN * kFK * 2;        // 32 KB B tile per stage
constexpr int kFThreads = 320;                 // producer, MMA, 4 epilogue warps, 4 pre-decode warps
constexpr uint32_t kFTmem = 2 * kFN;           // two fp32 accumulators
constexpr uint32_t kRBox = 32 * 64 * 2;        // one 32-row x 64-class bf16 output box
constexpr int kMaxNT = 8;

__device__ __forceinline__ uint32_t mapa_u32(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_async_v2(uint32_t raddr, float x, float y, uint32_t rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(raddr),
               "f"(x), "f"(y), "r"(rbar)
               : "memory");
}
__device__ __forceinline__ bool try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool wait_cluster(uint64_t* bar, uint32_t parity, int* status) {
  if (try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 0; it < kWaitMaxIters; ++it) {
    if (try_wait_cluster(bar, parity)) return true;
    if ((it & 63u) == 63u && globaltimer_ns() - t0 > kWaitMaxNs) break;
  }
  atomicOr(status, kErrWaitTimeout);
  return false;
}
__device__ __forceinline__ void mbar_arrive_remote(uint32_t rbar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(rbar) : "memory");
}
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

struct FusedSmem {
  uint32_t sA, sB, box, stats, bars, total;
};
// The decode plan of the early decode terms, for at most kPreMaxDev stores
// whose coefficient deviates (CR: the stragglers).
struct PrePlan {
  float B;
  int ndev;
  int dev[kPreMaxDev];
  float devc[kPreMaxDev];
};
__host__ __device__ inline FusedSmem fused_smem(int NT) {
  FusedSmem s;
  s.sA = 0;
  s.sB = kFStages * kFA;
  s.box = s.sB + kFStages * kFB;
  s.stats = s.box + 4 * kRBox;
  s.bars = s.stats + 2 * NT * kFM * 8;
  s.total = s.bars + 32 * 8;
  return s;
}

}  // namespace

__global__ void __launch_bounds__(kFThreads, 1)
tc_logits_softmax_kernel(const __grid_constant__ CUtensorMap tmXq, const __grid_constant__ CUtensorMap tmW,
                         const __grid_constant__ CUtensorMap tmR, TcSoftmaxParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ PrePlan pre_plan;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int NT = p.NT;
  const FusedSmem L = fused_smem(NT);
  uint8_t* sA = sm + L.sA;
  uint8_t* sB = sm + L.sB;
  uint8_t* sBox = sm + L.box;
  float2* stats = reinterpret_cast<float2*>(sm + L.stats);   // [2][NT][128] (max, sum) per source CTA and row
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L.bars);
  uint64_t* full = bars + 0;          // [4]
  uint64_t* empty = bars + 4;         // [4]
  uint64_t* acc_full = bars + 8;      // [2]
  uint64_t* acc_empty = bars + 10;    // [2]
  uint64_t* stats_full = bars + 12;   // [2] every CTA's (max, sum) of the tile's rows arrived
  uint64_t* stats_empty = bars + 14;  // [2] every epilogue warp of the cluster has read them
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);
  int* cta_err = reinterpret_cast<int*>(bars + 17);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = (int)cluster_rank();
  const uint16_t all_mask = (uint16_t)((1u << NT) - 1u);
  const int part = kFM / NT;                               // A rows each CTA loads and multicasts
  const int ncl = (int)gridDim.x / NT, cid = (int)blockIdx.x / NT;
  const int my_tiles = p.ntiles > cid ? (p.ntiles - cid + ncl - 1) / ncl : 0;

  if (threadIdx.x == 0) {
    *cta_err = 0;
    for (int s = 0; s < kFStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], NT);          // every CTA's MMAs read the stage (its A part is everyone's)
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);
      mbar_init(&stats_full[a], 1);
      mbar_init(&stats_empty[a], 4 * NT);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kFTmem)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 64) {
    // the row statistics of the first two tiles may arrive before this CTA reaches them
    for (int a = 0; a < 2 && a < my_tiles; ++a) mbar_arrive_expect_tx(&stats_full[a], (uint32_t)NT * kFM * 8);
  }
  tc_fence_before();
  cluster_sync_all();                    // peers' barriers exist before any multicast or st.async
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (threadIdx.x == 0) grid_dep_launch();

  if (warp == 0 && lane == 0) {
    // ---- producer ----------------------------------------------------------
    grid_dep_wait();                     // W is the previous step's update
    int it = 0;
    bool ok = true;
    for (int i = 0; i < my_tiles && ok; ++i) {
      const int4 tl = p.tiles[cid + i * ncl];
      for (int kb = 0; kb < p.nk; ++kb, ++it) {
        const int s = it % kFStages;
        if (it >= kFStages && !mbar_wait(&empty[s], ((it / kFStages) - 1) & 1, p.status)) { ok = false; break; }
        mbar_arrive_expect_tx(&full[s], kFA + kFB);
        tma_load_2d_mc(sA + s * kFA + rank * part * 128, &tmXq, kb * kFK, tl.x + rank * part, &full[s], all_mask);
        for (int j = 0; j < 2; ++j)
          tma_load_2d(sB + s * kFB + j * (kFB / 2), &tmW, kb * kFK, rank * kFN + j * (kFN / 2), &full[s]);
      }
    }
    if (!ok) atomicExch(cta_err, 1);
    for (int s = 0; s < kFStages && s < it; ++s) {
      const int last = ((it - 1 - s) / kFStages) * kFStages + s;
      mbar_wait(&full[s], (last / kFStages) & 1, p.status);
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer ----------------------------------------------------------
    constexpr uint32_t idesc = idesc_bf16_f32(kFM, kFN, false, false);
    int it = 0;
    bool ok = true;
    for (int i = 0; i < my_tiles && ok; ++i) {
      const int acc = i & 1;
      if (i >= 2 && !mbar_wait(&acc_empty[acc], ((i / 2) - 1) & 1, p.status)) { ok = false; break; }
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(acc * kFN);
      for (int kb = 0; kb < p.nk; ++kb, ++it) {
        const int s = it % kFStages;
        if (!mbar_wait(&full[s], (it / kFStages) & 1, p.status)) { ok = false; break; }
        tc_fence_after();
        const uint64_t da = smem_desc_sw128(smem_u32(sA + s * kFA), 16, 1024);
        const uint64_t db = smem_desc_sw128(smem_u32(sB + s * kFB), 16, 1024);
        umma_bf16(d, da, db, idesc, kb != 0 ? 1u : 0u);
        umma_bf16(d, da + 2, db + 2, idesc, 1u);
        umma_bf16(d, da + 4, db + 4, idesc, 1u);
        umma_bf16(d, da + 6, db + 6, idesc, 1u);
        umma_commit_mc(&empty[s], all_mask);   // released in every CTA's count
      }
      if (!ok) break;
      umma_commit(&acc_full[acc]);
    }
    if (!ok) atomicExch(cta_err, 1);
  } else if (warp >= 6) {
    // ---- pre-decode: the part of the step's decode that reads only data the
    // step leaves as it is (§V-B decode with the slot-total form): for this
    // CTA's slice of the float4 columns, pre = B sum_{o != o_t} U[o] +
    // sum_{stores r with b_r != B} (b_r - B) sum_{o != o_t} store[r][o].  It
    // streams beside the GEMM, so the decode after the gradient contraction
    // reads only pre, U[o_t] and the deviating stores' slot o_t.
    if (p.pre_out) {
      const DecodeArgs& a = p.pre;
      if (warp == 6) derive_plan_warp(a, pre_plan, lane);   // needs only the mask
      asm volatile("bar.sync 1, 128;" ::: "memory");          // the four pre-decode warps
      grid_dep_wait();                   // the stores and slot totals of the previous steps
      const int64_t P4 = a.P / 4, slotP = (int64_t)a.c * P4;
      const int c = a.c, sl = a.slot;
      const int64_t q0 = P4 * blockIdx.x / gridDim.x, q1 = P4 * (blockIdx.x + 1) / gridDim.x;
      const float4* U = reinterpret_cast<const float4*>(a.U);
      const float4* store = reinterpret_cast<const float4*>(a.store);
      for (int64_t pc = q0 + (threadIdx.x - 192); pc < q1; pc += 128) {
        float4 V = f4zero(), D = f4zero();
        for (int o0 = 0; o0 < c; o0 += 8) {
          float4 v[8];
#pragma unroll
          for (int j = 0; j < 8; ++j)
            v[j] = (o0 + j < c && o0 + j != sl) ? __ldcg(U + (int64_t)(o0 + j) * P4 + pc) : f4zero();
#pragma unroll
          for (int j = 0; j < 8; ++j) V = f4add(V, v[j]);
        }
        for (int q = 0; q < pre_plan.ndev; ++q) {
          const float4* base = store + (int64_t)pre_plan.dev[q] * slotP + pc;
          float4 Cr = f4zero();
          for (int o0 = 0; o0 < c; o0 += 8) {
            float4 v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = (o0 + j < c && o0 + j != sl) ? __ldcg(base + (int64_t)(o0 + j) * P4) : f4zero();
#pragma unroll
            for (int j = 0; j < 8; ++j) Cr = f4add(Cr, v[j]);
          }
          D = f4fma(pre_plan.devc[q], Cr, D);
        }
        reinterpret_cast<float4*>(p.pre_out)[pc] = f4fma(pre_plan.B, V, D);
      }
    }
  } else if (warp >= 2) {
    // ---- epilogue: softmax residual of this CTA's 256 classes ---------------
    const int q = warp & 3;
    const int t = threadIdx.x - 64;
    const int row = q * 32 + lane;                           // tile row of this thread
    uint8_t* box = sBox + (warp - 2) * kRBox;
    grid_dep_wait();                     // R and the slot total are read by the previous step until now
    if (p.zero_buf) {
      const int64_t nthr = (int64_t)gridDim.x * 128, tid = (int64_t)blockIdx.x * 128 + t;
      for (int64_t k = tid; k < p.zero_n4; k += nthr)
        reinterpret_cast<float4*>(p.zero_buf)[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const uint32_t stats_base = smem_u32(stats);
    const int cls0 = rank * kFN;
    bool ok = true;
    int nbox = 0;
    for (int i = 0; i < my_tiles && ok; ++i) {
      const int acc = i & 1, par = i & 1;
      const int4 tl = p.tiles[cid + i * ncl];
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[acc], (i / 2) & 1, p.status))) { ok = false; break; }
      tc_fence_after();
      const uint32_t t_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kFN);
      // pass 1: running max and sum of exp over this CTA's classes
      float m = -INFINITY, ssum = 0.f;
      for (int ch = 0; ch < kFN / 32; ++ch) {
        const int c0 = cls0 + ch * 32;
        if (c0 >= p.K) break;                                // warp-uniform
        uint32_t r[32];
        tmem_ld32(t_base + ch * 32, r);
        tmem_ld_wait();
        float mc = -INFINITY;
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (c0 + c < p.K) mc = fmaxf(mc, __uint_as_float(r[c]));
        if (mc > m) {
          ssum = m == -INFINITY ? 0.f : ssum * __expf(m - mc);
          m = mc;
        }
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (c0 + c < p.K) ssum += __expf(__uint_as_float(r[c]) - m);
      }
      // every CTA of the cluster gets this row's (max, sum) of this CTA's classes,
      // once all of them have read what this CTA sent two tiles ago
      if (i >= 2 && !__all_sync(0xffffffffu, wait_cluster(&stats_empty[par], ((i / 2) - 1) & 1, p.status))) {
        ok = false;
        break;
      }
      const uint32_t local = stats_base + (uint32_t)(((par * NT + rank) * kFM + row) * 8);
      const uint32_t lbar = smem_u32(&stats_full[par]);
      for (int dst = 0; dst < NT; ++dst) st_async_v2(mapa_u32(local, dst), m, ssum, mapa_u32(lbar, dst));
      if (!__all_sync(0xffffffffu, wait_cluster(&stats_full[par], (i / 2) & 1, p.status))) { ok = false; break; }
      float M = -INFINITY;
      for (int j = 0; j < NT; ++j) M = fmaxf(M, stats[(par * NT + j) * kFM + row].x);
      float S = 0.f;
      for (int j = 0; j < NT; ++j) {
        const float2 v = stats[(par * NT + j) * kFM + row];
        if (v.x != -INFINITY) S += v.y * __expf(v.x - M);
      }
      __syncwarp();
      if (i + 2 < my_tiles) {
        if (t == 0) mbar_arrive_expect_tx(&stats_full[par], (uint32_t)NT * kFM * 8);
        if (lane == 0)
          for (int dst = 0; dst < NT; ++dst) mbar_arrive_remote(mapa_u32(smem_u32(&stats_empty[par]), dst));
      }
      const bool valid = row < tl.z;
      const int lab = valid ? p.y[tl.x + row] - cls0 : -1;   // label's column in this CTA's 256
      const float inv = 1.0f / S;
      // pass 2: residuals, 64 classes per TMA-stored box
      for (int pr = 0; pr < kFN / 64 && cls0 + pr * 64 < p.K; ++pr) {   // boxes past K stay zero
        if (lane == 0 && nbox > 0) bulk_wait_read0();
        __syncwarp();
        uint4* rowp = reinterpret_cast<uint4*>(box + lane * 128);
        for (int h = 0; h < 2; ++h) {
          uint32_t r[32];
          tmem_ld32(t_base + (pr * 2 + h) * 32, r);
          tmem_ld_wait();
          const int cb = pr * 64 + h * 32;                   // column within this CTA's 256
          uint32_t w[16];
#pragma unroll
          for (int c = 0; c < 32; c += 2) {
            float v0 = 0.f, v1 = 0.f;
            if (valid && cls0 + cb + c < p.K)
              v0 = __expf(__uint_as_float(r[c]) - M) * inv - (cb + c == lab ? 1.f : 0.f);
            if (valid && cls0 + cb + c + 1 < p.K)
              v1 = __expf(__uint_as_float(r[c + 1]) - M) * inv - (cb + c + 1 == lab ? 1.f : 0.f);
            w[c / 2] = pack_bf16(v0, v1);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
            rowp[(h * 4 + u) ^ (lane & 7)] = make_uint4(w[4 * u], w[4 * u + 1], w[4 * u + 2], w[4 * u + 3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&tmR, box, cls0 + pr * 64, tl.y + q * 32);
          bulk_commit();
        }
        ++nbox;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
    if (!ok) atomicExch(cta_err, 1);
  }
  __syncthreads();
  tc_fence_before();
  cluster_sync_all();                    // no multicast, st.async or remote arrive is still aimed at this CTA
  tc_fence_after();
  if (warp == 1) {
    if (*cta_err && lane == 0) {
      // the MMAs already issued finish before TMEM is released
      for (int a = 0; a < 2 && a < my_tiles; ++a) {
        const int last = ((my_tiles - 1 - a) / 2) * 2 + a;
        mbar_wait(&acc_full[a], (last / 2) & 1, p.status);
      }
    }
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kFTmem) : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
static size_t fused_smem_bytes(int NT) { return 1024 + fused_smem(NT).total; }

static cudaError_t fused_attributes(int NT) {
  // clusters of at most 8 CTAs (kMaxNT): the portable size, no opt-in needed
  return cudaFuncSetAttribute(tc_logits_softmax_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)fused_smem_bytes(NT));
}

int tc_softmax_max_clusters(int NT) {
  if (NT < 1 || NT > kMaxNT || (kFM % NT) != 0 || (NT & (NT - 1)) != 0) return 0;
  if (fused_attributes(NT) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(NT);
  cfg.blockDim = dim3(kFThreads);
  cfg.dynamicSmemBytes = fused_smem_bytes(NT);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = NT;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int nc = 0;
  if (cudaOccupancyMaxActiveClusters(&nc, tc_logits_softmax_kernel, &cfg) != cudaSuccess) return 0;
  return nc;
}

cudaError_t launch_tc_softmax(const void* tmXq, const void* tmW, const void* tmR, const TcSoftmaxParams& p,
                              int nclusters, cudaStream_t st) {
  if (p.ntiles <= 0) return cudaSuccess;
  if (nclusters < 1 || p.NT < 1 || p.NT > kMaxNT) return cudaErrorInvalidValue;
  cudaError_t e = fused_attributes(p.NT);
  if (e != cudaSuccess) return e;
  const int ncl = nclusters < p.ntiles ? nclusters : p.ntiles;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(ncl * p.NT));
  cfg.blockDim = dim3(kFThreads);
  cfg.dynamicSmemBytes = fused_smem_bytes(p.NT);
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.NT;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pdl ? 2 : 1;
  CUtensorMap a, b, r;
  std::memcpy(&a, tmXq, sizeof(CUtensorMap));
  std::memcpy(&b, tmW, sizeof(CUtensorMap));
  std::memcpy(&r, tmR, sizeof(CUtensorMap));
  return cudaLaunchKernelEx(&cfg, tc_logits_softmax_kernel, a, b, r, p);
}

}  // namespace pgc
