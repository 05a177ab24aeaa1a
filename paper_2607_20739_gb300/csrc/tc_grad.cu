// Gradient contraction of the tensor-core softmax path (§III with f = log
// sum_k exp(w_k.x) - w_y.x): for every evaluated partition e,
//
//   G_e[k][j] = (1/m_e) sum_{r in D_e} R[r][k] X[r][j]     A = R (MN-major), B = X (MN-major)
//
// written straight into every store that keeps the partition, and, in steady
// steps, the slot total U[o_t] = sum_e G_e (§V-B) formed on the way out.
//
// Work is split into units {pair tile, run of partitions}: a cluster of two
// CTAs owns the 256 x 256 output tile (class tiles 2mp, 2mp+1; feature tile
// nt) for a run of up to eight partitions and computes G_e of each in turn.
// Each CTA loads its 128 x 64 R tile and one half of the 64 x 256 X tile,
// multicast into both CTAs, into a 4-stage ring (2-D TMA, 128-byte swizzle);
// warp 1 issues tcgen05.mma (M = 128 classes, N = 256 features, K = 16 rows)
// into one of two TMEM accumulators.  Eight epilogue warps (two per TMEM lane
// quarter, 128 columns each) drain the other, 32 x 32 blocks at a time: a
// block is written row-per-lane into the warp's 128-byte-swizzled box, which
// one lane sends by TMA tensor store (evict-first: the stores are only read
// back for stragglers) into every store that keeps the partition; the box is
// rewritten once those copies have read it.  Each thread also keeps its row's
// share of the run's sum in registers, added into U[o_t] with one TMA
// reduce-add per block at the end of the run.  So U costs one reduce per run
// instead of one per partition.
// Every wait is bounded; the TMEM allocation is released on every path.
//
// Pair form (kPair, the default): the same units and epilogue, but the
// pair's MMA is one tcgen05.mma.cta_group::2 (M = 256 classes: 128 from each
// CTA's TMEM and shared memory; N = 256 features: each CTA holds 128 of them)
// issued by the even CTA.  A stage then holds 16 KB of R and 16 KB of X per
// CTA instead of 16 + 32, so six stages fit where four did; each CTA's TMA
// loads complete on the even CTA's stage barrier, and the MMA's commits free
// the stage and hand over the accumulator in both CTAs.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdlib>
#include <cstring>

#include "tc_common.cuh"

namespace pgc {

namespace {

constexpr int kGM = 128, kGN = 256, kGK = 64;
constexpr uint32_t kGA = kGM * kGK * 2;         // 16 KB R tile (two 64 x 64 boxes)
// per CTA: stages, and the X tile it holds (all 256 features, multicast
// halves; or, in the pair form, its 128 of them)
template <bool kPair> struct GradCfg {
  static constexpr int kStages = kPair ? 6 : 4;
  static constexpr uint32_t kB = (kPair ? kGN / 2 : kGN) * kGK * 2;   // 16 or 32 KB
};
constexpr int kGThreads = 320;                  // producer, MMA, 8 epilogue warps
constexpr int kGEpi = 8;
constexpr uint32_t kGTmem = 2 * kGN;            // two fp32 accumulators
constexpr uint32_t kGBox = 32 * 32 * 4;         // one 32 x 32 fp32 output box

struct GradSmem {
  uint32_t sA, sB, box, bars, total;
};
template <bool kPair>
__host__ __device__ constexpr GradSmem grad_smem() {
  constexpr int S = GradCfg<kPair>::kStages;
  constexpr uint32_t B = GradCfg<kPair>::kB;
  return GradSmem{0, S * kGA, S * (kGA + B), S * (kGA + B) + kGEpi * kGBox, S * (kGA + B) + kGEpi * kGBox + 24 * 8};
}

__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

// stage 8 values (columns 8 qt .. 8 qt + 7) of this lane's row into its
// 128-byte row of a swizzled box (16-byte chunk c at c ^ (row & 7))
__device__ __forceinline__ void stage_quarter(uint8_t* box, int lane, int qt, const float* v) {
  float4* rowp = reinterpret_cast<float4*>(box + lane * 128);
  rowp[(2 * qt) ^ (lane & 7)] = make_float4(v[0], v[1], v[2], v[3]);
  rowp[(2 * qt + 1) ^ (lane & 7)] = make_float4(v[4], v[5], v[6], v[7]);
}

}  // namespace

// Ten warps put three on some of the SM's four register-file quarters, so a
// thread gets at most 168 registers; the epilogue keeps 128 partial sums of
// the slot total in them and reads TMEM 16 columns at a time.
template <bool kPair>
__global__ void __launch_bounds__(kGThreads, 1)
tc_grad_kernel(const __grid_constant__ CUtensorMap tmR, const __grid_constant__ CUtensorMap tmX,
               const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmS, TcGradParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int kGS = GradCfg<kPair>::kStages;
  constexpr uint32_t kGB = GradCfg<kPair>::kB;
  constexpr GradSmem L = grad_smem<kPair>();
  uint8_t* sA = sm + L.sA;
  uint8_t* sB = sm + L.sB;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L.bars);
  uint64_t* full = bars;                // [kGS]
  uint64_t* empty = bars + kGS;         // [kGS]
  uint64_t* acc_full = bars + 2 * kGS;  // [2]
  uint64_t* acc_empty = acc_full + 2;   // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 4);
  int* cta_err = reinterpret_cast<int*>(acc_full + 5);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = (int)cluster_rank();
  constexpr uint16_t kBoth = 0x3;
  // pair form: the even CTA issues the MMAs and owns the stage and
  // accumulator barriers they wait on
  const bool issuer = !kPair || rank == 0;
  if (threadIdx.x == 0) {
    *cta_err = 0;
    for (int s = 0; s < kGS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kPair ? 1 : 2);   // the pair MMA's commit, or the MMAs of both CTAs
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], kPair ? 2 * kGEpi : kGEpi);   // pair form: both CTAs' epilogues
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (kPair) {
      // one warp of each CTA of the pair allocates, together
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                   "r"(kGTmem)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                   "r"(kGTmem)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  tc_fence_before();
  cluster_sync_all();                    // the peer's barriers exist before any multicast
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (threadIdx.x == 0) grid_dep_launch();
  if (p.pdl) grid_dep_wait();           // R is the previous kernel's output; U was zeroed there

  const int pair = (int)blockIdx.x >> 1, npairs = (int)gridDim.x >> 1;
  const int my_units = p.nunits > pair ? (p.nunits - pair + npairs - 1) / npairs : 0;

  if (warp == 0 && lane == 0) {
    // ---- producer ----------------------------------------------------------
    int it = 0;
    bool ok = true;
    for (int i = 0; i < my_units && ok; ++i) {
      const int4 u = p.units[pair + i * npairs];
      const int mt = 2 * u.x + rank, nt = u.y;
      for (int j = 0; j < u.w && ok; ++j) {
        const int b = u.z + j;
        const int nkb = p.nk[b];
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kGS;
          if (it >= kGS && !mbar_wait(&empty[s], ((it / kGS) - 1) & 1, p.status)) { ok = false; break; }
          uint8_t* a_dst = sA + (size_t)s * kGA;
          uint8_t* b_dst = sB + (size_t)s * kGB;
          if constexpr (kPair) {
            // this CTA's R rows and its 128 features of X, counted on the
            // even CTA's stage barrier (which expects both CTAs' bytes)
            if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * (kGA + kGB));
            const uint32_t fb = cluster_addr(&full[s], 0);
            for (int q = 0; q < 2; ++q)
              tma_load_2d_pair(a_dst + q * 8192, &tmR, mt * kGM + q * 64, p.a_off[b] + kb * kGK, fb);
            for (int q = 0; q < 2; ++q)
              tma_load_2d_pair(b_dst + q * 8192, &tmX, nt * kGN + rank * 128 + q * 64, p.b_off[b] + kb * kGK, fb);
          } else {
            mbar_arrive_expect_tx(&full[s], kGA + kGB);
            for (int q = 0; q < 2; ++q)
              tma_load_2d(a_dst + q * 8192, &tmR, mt * kGM + q * 64, p.a_off[b] + kb * kGK, &full[s]);
            for (int q = 2 * rank; q < 2 * rank + 2; ++q)
              tma_load_2d_mc(b_dst + q * 8192, &tmX, nt * kGN + q * 64, p.b_off[b] + kb * kGK, &full[s], kBoth);
          }
        }
      }
    }
    if (!ok) atomicExch(cta_err, 1);
    // no copy may outlive the CTA: wait for the last fill of every stage
    // (pair form: the last MMA commit on a stage follows both CTAs' copies)
    for (int s = 0; s < kGS && s < it; ++s) {
      const int last = ((it - 1 - s) / kGS) * kGS + s;
      if (kPair) mbar_wait(&empty[s], (last / kGS) & 1, p.status);
      else mbar_wait(&full[s], (last / kGS) & 1, p.status);
    }
  } else if (warp == 1 && lane == 0 && issuer) {
    // ---- MMA issuer --------------------------------------------------------
    constexpr uint32_t idesc = idesc_bf16_f32(kPair ? 2 * kGM : kGM, kGN, true, true);
    int it = 0, tt = 0;
    bool ok = true;
    for (int i = 0; i < my_units && ok; ++i) {
      const int4 u = p.units[pair + i * npairs];
      for (int j = 0; j < u.w && ok; ++j, ++tt) {
        const int acc = tt & 1;
        if (tt >= 2 && !mbar_wait(&acc_empty[acc], ((tt / 2) - 1) & 1, p.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem + (uint32_t)(acc * kGN);
        const int nkb = p.nk[u.z + j];
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kGS;
          if (!mbar_wait(&full[s], (it / kGS) & 1, p.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a_base = smem_u32(sA + (size_t)s * kGA);
          const uint32_t b_base = smem_u32(sB + (size_t)s * kGB);
#pragma unroll
          for (int kk = 0; kk < kGK / 16; ++kk) {
            // MN-major: the next 16 K rows are two 8-row groups (2 KB) further
            const uint64_t da = smem_desc_sw128(a_base + kk * 2048, 8192, 1024);
            const uint64_t db = smem_desc_sw128(b_base + kk * 2048, 8192, 1024);
            if constexpr (kPair) umma_bf16_pair(d_tmem, da, db, idesc, (kb | kk) != 0 ? 1u : 0u);
            else umma_bf16(d_tmem, da, db, idesc, (kb | kk) != 0 ? 1u : 0u);
          }
          // the stage is free again, in both CTAs
          if constexpr (kPair) umma_commit_pair_mc(&empty[s], kBoth);
          else umma_commit_mc(&empty[s], kBoth);
        }
        if (!ok) break;
        // the accumulator is complete (pair form: in both CTAs)
        if constexpr (kPair) umma_commit_pair_mc(&acc_full[acc], kBoth);
        else umma_commit(&acc_full[acc]);
      }
    }
    if (!ok) atomicExch(cta_err, 1);
  } else if (warp >= 2) {
    // ---- epilogue ----------------------------------------------------------
    // Warp w drains TMEM lanes 32q..32q+31 (q = w % 4: the lane quarter it may
    // read), columns 128h..128h+127, 32 at a time, into its 32 x 32 box of
    // shared memory laid out as the 128-byte-swizzled TMA box (16-byte chunk
    // c of row r at chunk c ^ (r & 7)); lane 0 stores it.  The box is
    // rewritten only after the previous bulk group has finished reading it.
    const int q = warp & 3, h = (warp - 2) >> 2;
    uint8_t* box = sm + L.box + (size_t)(warp - 2) * kGBox;
    bool pending = false;
    int tt = 0;
    bool ok = true;
    float usum[4][32];
    for (int i = 0; i < my_units && ok; ++i) {
      const int4 u = p.units[pair + i * npairs];
      const int mt = 2 * u.x + rank, nt = u.y;
      const int row0 = mt * kGM + q * 32;              // first class of this warp's rows
      const bool rows_exist = row0 < p.m_limit;        // warp-uniform
      const int n0 = nt * kGN + h * 128;               // first feature of this warp's columns
#pragma unroll
      for (int ch = 0; ch < 4; ++ch)
#pragma unroll
        for (int c = 0; c < 32; ++c) usum[ch][c] = 0.f;
      for (int j = 0; j < u.w; ++j, ++tt) {
        const int b = u.z + j;
        const int acc = tt & 1;
        if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[acc], (tt / 2) & 1, p.status))) { ok = false; break; }
        tc_fence_after();
        const float sc = p.scale[b];
        const uint32_t t_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kGN + h * 128);
        const int32_t* dl = p.dest + (int64_t)b * p.ndest;
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          if (rows_exist && pending) {             // the last U reduce-add has read the box
            if (lane == 0) bulk_wait_read0();
            __syncwarp();
            pending = false;
          }
#pragma unroll
          for (int qt = 0; qt < 4; ++qt) {
            uint32_t r[8];
            tmem_ld8(t_base + ch * 32 + qt * 8, r);
            tmem_ld_wait();
            float* g = reinterpret_cast<float*>(r);
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              g[c] = sc * __uint_as_float(r[c]);
              usum[ch][8 * qt + c] += g[c];
            }
            if (rows_exist) stage_quarter(box, lane, qt, g);
          }
          if (rows_exist) {
            // the box goes to every store keeping the copy by TMA (rows past
            // the class count are outside the map and dropped); it is
            // rewritten only after these copies have read it
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              const uint64_t pol = policy_evict_first();
              for (int k = 0; k < p.ndest; ++k) {
                const int dd = dl[k];
                if (dd >= 0) tma_store_3d_hint(&tmS, box, n0 + ch * 32, row0, dd, pol);
              }
              bulk_commit();
            }
            pending = true;
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (kPair && rank != 0) mbar_arrive_cluster(cluster_addr(&acc_empty[acc], 0));
          else mbar_arrive(&acc_empty[acc]);
        }
      }
      if (ok && p.u_reduce && rows_exist) {
        // this run's share of the slot total
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          if (lane == 0 && pending) bulk_wait_read0();
          __syncwarp();
#pragma unroll
          for (int qt = 0; qt < 4; ++qt) stage_quarter(box, lane, qt, &usum[ch][8 * qt]);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_reduce_add_3d_hint(&tmU, box, n0 + ch * 32, row0, p.u_slot, policy_evict_last());
            bulk_commit();
          }
          pending = true;
        }
      }
    }
    if (lane == 0) bulk_wait_all();      // stores done before the CTA exits
    __syncwarp();
    if (!ok) atomicExch(cta_err, 1);
  }
  __syncthreads();
  if (warp == 1 && lane == 0 && issuer && *cta_err) {
    // every MMA has completed before its accumulator was drained; after a
    // failure, wait (bounded) for the last commits before TMEM is released
    int total = 0;
    for (int i = 0; i < my_units; ++i) total += p.units[pair + i * npairs].w;
    for (int a = 0; a < 2 && a < total; ++a) {
      const int last = ((total - 1 - a) / 2) * 2 + a;
      mbar_wait(&acc_full[a], (last / 2) & 1, p.status);
    }
  }
  __syncthreads();
  cluster_sync_all();                    // no multicast, MMA or remote arrive is still aimed at this CTA
  if (warp == 1) {
    tc_fence_after();
    if constexpr (kPair)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kGTmem) : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kGTmem) : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
template <bool kPair>
static size_t grad_smem_bytes() { return 1024 + grad_smem<kPair>().total; }

// The pair form unless PGC_GRAD_PAIR_MMA=0 asks for the two-MMA form.
static bool use_pair_mma() {
  static int v = -1;
  if (v < 0) {
    const char* env = std::getenv("PGC_GRAD_PAIR_MMA");
    v = (env && env[0] == '0') ? 0 : 1;
  }
  return v != 0;
}

template <bool kPair>
static int max_pairs() {
  const size_t smem = grad_smem_bytes<kPair>();
  if (cudaFuncSetAttribute(tc_grad_kernel<kPair>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess)
    return 0;
  cudaLaunchConfig_t q = {};
  q.gridDim = dim3(2);
  q.blockDim = dim3(kGThreads);
  q.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  q.attrs = attr;
  q.numAttrs = 1;
  int nc = 0;
  if (cudaOccupancyMaxActiveClusters(&nc, tc_grad_kernel<kPair>, &q) != cudaSuccess) return 0;
  return nc;
}

int tc_grad_max_pairs() {
  static int mp = -1;
  if (mp < 0) mp = use_pair_mma() ? max_pairs<true>() : max_pairs<false>();
  return mp;
}

cudaError_t launch_tc_grad(const void* tmR, const void* tmX, const void* tmU, const void* tmS, const TcGradParams& p,
                           int npairs, cudaStream_t st) {
  if (p.nunits <= 0) return cudaSuccess;
  if (npairs < 1) return cudaErrorInvalidValue;
  const bool pair_mma = use_pair_mma();
  const size_t smem = pair_mma ? grad_smem_bytes<true>() : grad_smem_bytes<false>();
  cudaError_t e = pair_mma
                      ? cudaFuncSetAttribute(tc_grad_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)
                      : cudaFuncSetAttribute(tc_grad_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int pairs = npairs < p.nunits ? npairs : p.nunits;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(2 * pairs));
  cfg.blockDim = dim3(kGThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pdl ? 2 : 1;
  CUtensorMap a, b, u, w;
  std::memcpy(&a, tmR, sizeof(CUtensorMap));
  std::memcpy(&b, tmX, sizeof(CUtensorMap));
  std::memcpy(&u, tmU, sizeof(CUtensorMap));
  std::memcpy(&w, tmS, sizeof(CUtensorMap));
  return pair_mma ? cudaLaunchKernelEx(&cfg, tc_grad_kernel<true>, a, b, u, w, p)
                  : cudaLaunchKernelEx(&cfg, tc_grad_kernel<false>, a, b, u, w, p);
}

}  // namespace pgc
