// Logits GEMM of the tensor-core softmax path (§III with f = log sum_k
// exp(w_k.x) - w_y.x) for class counts whose 256-class tiles do not form a
// cluster of 1, 2, 4 or 8 CTAs (the fused kernel covers those):
//
//   Z[r][k] = sum_j X[r][j] W[k][j]       A = X (K-major), B = W (K-major)
//
// followed by the residual kernel R = softmax(Z) - onehot(y).  One
// persistent, warp-specialised kernel launched as clusters of two CTAs: the
// pair computes the row tiles 2i and 2i+1 of the same (batch, class tile), so
// the B tile is common; each CTA loads its own 128x64 A tile and one 128-row
// half of the 256x64 B tile, multicast into both CTAs, into a 4-stage
// shared-memory ring with 2-D TMA (cp.async.bulk.tensor, 128-byte swizzle).
// A stage is refilled once the MMAs of both CTAs have read it.  Warp 1 issues
// tcgen05.mma.cta_group::1.kind::f16 (bf16 in, fp32 accumulate) into one of
// two 128x256 TMEM accumulators, and warps 2-5 drain the other accumulator
// with tcgen05.ld, stage 32 x 32 fp32 boxes in (swizzled) shared memory and
// write them to Z with TMA stores.
// Every wait is bounded; the TMEM allocation is released on every path.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "tc_common.cuh"

namespace pgc {

constexpr int kTM = 128, kTN = 256, kTK = 64;
constexpr int kGStages = 4;
constexpr uint32_t kABytes = kTM * kTK * 2;    // 16 KB
constexpr uint32_t kBBytes = kTN * kTK * 2;    // 32 KB
constexpr int kGemmThreads = 192;              // producer, MMA, 4 epilogue warps
constexpr uint32_t kTmemCols = 2 * kTN;        // two fp32 accumulators
constexpr uint32_t kStageBox = 32 * 32 * 4;    // one 32 x 32 fp32 output box
constexpr uint32_t kEpiBytes = 4 * 2 * kStageBox;  // two boxes per epilogue warp

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------
// Pair tile t -> batch b, N tile nt and this CTA's M tile mt = 2 mp + rank;
// false when mt is past the batch's M tiles (odd count: the CTA computes a
// dummy tile to keep the pair in step and stores nothing).
__device__ __forceinline__ bool decode_tile(const TcGemmParams& p, int t, int rank, int& b, int& mt, int& nt) {
  int lo = 0, hi = p.nbatch - 1;
  while (lo < hi) {                      // last b with tile_prefix[b] <= t
    const int mid = (lo + hi + 1) >> 1;
    if (p.tile_prefix[mid] <= t) lo = mid; else hi = mid - 1;
  }
  b = lo;
  const int rem = t - p.tile_prefix[b];
  mt = 2 * (rem / p.NT) + rank;
  nt = rem % p.NT;
  return mt < p.mt_count[b];
}

__global__ void __launch_bounds__(kGemmThreads, 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const __grid_constant__ CUtensorMap tmOut, TcGemmParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kGStages * kABytes;
  uint8_t* sE = sB + kGStages * kBBytes;          // epilogue boxes, 1024-byte aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(sE + kEpiBytes);
  uint64_t* empty = full + kGStages;
  uint64_t* acc_full = empty + kGStages;
  uint64_t* acc_empty = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  __shared__ int cta_err;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = (int)cluster_rank();
  constexpr uint16_t kPair = 0x3;
  if (threadIdx.x == 0) {
    cta_err = 0;
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 2);           // the MMAs of both CTAs read the stage
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cluster_sync_all();                    // the peer's barriers exist before any multicast
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (threadIdx.x == 0) grid_dep_launch();
  if (p.pdl) grid_dep_wait();           // inputs are the previous kernels' outputs

  // pair tiles of this cluster: pair, pair + npairs, ...
  const int pair = (int)blockIdx.x >> 1, npairs = (int)gridDim.x >> 1;
  const int my_tiles = p.total_tiles > pair ? (p.total_tiles - pair + npairs - 1) / npairs : 0;

  if (warp == 0 && lane == 0) {
    // ---- producer ----------------------------------------------------------
    int it = 0;
    bool ok = true;
    for (int i = 0; i < my_tiles && ok; ++i) {
      int b, mt, nt;
      decode_tile(p, pair + i * npairs, rank, b, mt, nt);
      const int nkb = p.nk[b];
      for (int kb = 0; kb < nkb; ++kb, ++it) {
        const int s = it % kGStages;
        // both CTAs' MMAs are done with the stage (this CTA's B half lands in both)
        if (it >= kGStages && !mbar_wait(&empty[s], ((it / kGStages) - 1) & 1, p.status)) { ok = false; break; }
        mbar_arrive_expect_tx(&full[s], kABytes + kBBytes);
        uint8_t* a_dst = sA + (size_t)s * kABytes;
        uint8_t* b_dst = sB + (size_t)s * kBBytes;
        tma_load_2d(a_dst, &tmA, kb * kTK, p.a_off[b] + mt * kTM, &full[s]);
        tma_load_2d_mc(b_dst + rank * (kBBytes / 2), &tmB, kb * kTK, nt * kTN + rank * (kTN / 2), &full[s], kPair);
      }
    }
    if (!ok) atomicExch(&cta_err, 1);
    // no copy may outlive the CTA: wait for the last fill of every stage
    for (int s = 0; s < kGStages && s < it; ++s) {
      const int last = ((it - 1 - s) / kGStages) * kGStages + s;
      mbar_wait(&full[s], (last / kGStages) & 1, p.status);
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer --------------------------------------------------------
    constexpr uint32_t idesc = idesc_bf16_f32(kTM, kTN, false, false);
    int it = 0;
    bool ok = true;
    for (int i = 0; i < my_tiles && ok; ++i) {
      int b, mt, nt;
      decode_tile(p, pair + i * npairs, rank, b, mt, nt);
      const int acc = i & 1;
      if (i >= 2 && !mbar_wait(&acc_empty[acc], ((i / 2) - 1) & 1, p.status)) { ok = false; break; }
      tc_fence_after();
      const uint32_t d_tmem = tmem + (uint32_t)(acc * kTN);
      const int nkb = p.nk[b];
      for (int kb = 0; kb < nkb; ++kb, ++it) {
        const int s = it % kGStages;
        if (!mbar_wait(&full[s], (it / kGStages) & 1, p.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t a_base = smem_u32(sA + (size_t)s * kABytes);
        const uint32_t b_base = smem_u32(sB + (size_t)s * kBBytes);
#pragma unroll
        for (int kk = 0; kk < kTK / 16; ++kk) {
          // K-major: the next 16 K elements are 32 bytes further along each
          // 128-byte row
          const uint64_t da = smem_desc_sw128(a_base + kk * 32, 16, 1024);
          const uint64_t db = smem_desc_sw128(b_base + kk * 32, 16, 1024);
          umma_bf16(d_tmem, da, db, idesc, (kb | kk) != 0 ? 1u : 0u);
        }
        umma_commit_mc(&empty[s], kPair);  // this CTA is done with the stage, in both CTAs' count
      }
      if (!ok) break;
      umma_commit(&acc_full[acc]);       // the accumulator is complete
    }
    if (!ok) atomicExch(&cta_err, 1);
  } else if (warp >= 2) {
    // ---- epilogue ----------------------------------------------------------
    // Warp q drains TMEM lanes 32q..32q+31 (tile rows), 32 columns at a time,
    // into a 32 x 32 box of shared memory laid out as the 128-byte-swizzled
    // TMA box (16-byte chunk j of row r at chunk j ^ (r & 7)), then lane 0
    // stores it.  Two boxes per warp alternate; a box is rewritten only after
    // the bulk group that read it has finished reading.
    const int q = warp & 3;              // TMEM lane quarter this warp may read
    uint8_t* box0 = sE + (size_t)(warp - 2) * 2 * kStageBox;
    int nbox = 0;
    for (int i = 0; i < my_tiles; ++i) {
      int b, mt, nt;
      const bool real = decode_tile(p, pair + i * npairs, rank, b, mt, nt);
      const int acc = i & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[acc], (i / 2) & 1, p.status))) {
        atomicExch(&cta_err, 1);
        break;
      }
      tc_fence_after();
      const int row0 = mt * kTM + q * 32;              // first tile row of this warp
      const bool rows_exist = real;
      const uint32_t t_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kTN);
      for (int ch = 0; ch < kTN / 32; ++ch) {
        uint32_t r[32];
        tmem_ld32(t_base + ch * 32, r);
        tmem_ld_wait();
        if (!rows_exist) continue;
        uint8_t* box = box0 + (nbox & 1) * kStageBox;
        if (lane == 0 && nbox >= 2) bulk_wait_read1();
        __syncwarp();
        float4* rowp = reinterpret_cast<float4*>(box + lane * 128);
#pragma unroll
        for (int v = 0; v < 8; ++v)
          rowp[v ^ (lane & 7)] = make_float4(__uint_as_float(r[4 * v]), __uint_as_float(r[4 * v + 1]),
                                             __uint_as_float(r[4 * v + 2]), __uint_as_float(r[4 * v + 3]));
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&tmOut, box, nt * kTN + ch * 32, (int)p.out_row0[b] + row0);
          bulk_commit();
        }
        ++nbox;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);
    }
    if (lane == 0) bulk_wait_all();      // stores done before the CTA exits
    __syncwarp();
  }
  __syncthreads();
  cluster_sync_all();                    // no multicast or remote arrive is still aimed at this CTA
  if (warp == 1) {
    // every MMA of this CTA has completed before its accumulator was drained;
    // after a failure, wait (bounded) for the last commits before releasing
    if (cta_err && lane == 0) {
      for (int a = 0; a < 2 && a < my_tiles; ++a) {
        const int last = ((my_tiles - 1 - a) / 2) * 2 + a;
        mbar_wait(&acc_full[a], (last / 2) & 1, p.status);
      }
    }
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor map: [outer][inner] row-major, row pitch in bytes,
// box {64, box_outer}, 128-byte swizzle; out-of-range elements read as zero.
bool make_tmap_bf16(void* tm_out, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
                    uint32_t box_outer) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_bytes};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(reinterpret_cast<CUtensorMap*>(tm_out), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_tmap_bf16_rows(void* tm_out, const void* base, uint64_t ld, uint64_t rows, uint32_t box_rows,
                         uint32_t box_blocks) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || ld % 64 != 0 || box_blocks < 1 || box_blocks > 256 || (ld / 64) % box_blocks != 0 || rows == 0)
    return false;
  alignas(64) CUtensorMap probe;
  CUtensorMap* out = tm_out ? reinterpret_cast<CUtensorMap*>(tm_out) : &probe;
  const void* b = base ? base : reinterpret_cast<const void*>(uintptr_t(1) << 20);
  cuuint64_t dims[3] = {64, rows, ld / 64};
  cuuint64_t strides[2] = {ld * 2, 128};
  cuuint32_t box[3] = {64, box_rows, box_blocks};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = fn(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(b), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_tmap_f32_box32(void* tm_out, const void* base, int rank, const uint64_t* dims, const uint64_t* strides) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || rank < 2 || rank > 3) return false;
  cuuint64_t d[3], st[2];
  cuuint32_t box[3] = {32, 32, 1}, estr[3] = {1, 1, 1};
  for (int i = 0; i < rank; ++i) d[i] = dims[i];
  for (int i = 0; i < rank - 1; ++i) st[i] = strides[i];
  const CUresult r = fn(reinterpret_cast<CUtensorMap*>(tm_out), CU_TENSOR_MAP_DATA_TYPE_FLOAT32, (cuuint32_t)rank,
                        const_cast<void*>(base), d, st, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

static size_t gemm_smem_bytes() {
  return 1024 + kGStages * (size_t)(kABytes + kBBytes) + kEpiBytes + sizeof(uint64_t) * (2 * kGStages + 4) + 16;
}

cudaError_t launch_tc_gemm(const void* tmA, const void* tmB, const void* tmOut, const TcGemmParams& p, int grid,
                           cudaStream_t st) {
  if (p.total_tiles <= 0) return cudaSuccess;
  auto kern = tc_gemm_kernel;
  const size_t smem = gemm_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kGemmThreads);
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
  // one pair per two SMs that can hold it at once
  static int mp = 0;
  if (mp == 0) {
    cudaLaunchConfig_t q = cfg;
    q.gridDim = dim3(2);
    q.numAttrs = 1;
    int nc = 0;
    e = cudaOccupancyMaxActiveClusters(&nc, kern, &q);
    if (e != cudaSuccess) return e;
    mp = nc > 0 ? nc : 1;
  }
  int pairs = grid / 2 < mp ? grid / 2 : mp;
  if (pairs > p.total_tiles) pairs = p.total_tiles;
  if (pairs < 1) pairs = 1;
  cfg.gridDim = dim3((unsigned)(2 * pairs));
  CUtensorMap a, b, o;
  std::memcpy(&a, tmA, sizeof(CUtensorMap));
  std::memcpy(&b, tmB, sizeof(CUtensorMap));
  std::memcpy(&o, tmOut, sizeof(CUtensorMap));
  return cudaLaunchKernelEx(&cfg, kern, a, b, o, p);
}

}  // namespace pgc
