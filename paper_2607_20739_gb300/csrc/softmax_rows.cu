// Softmax gradient for few classes (K <= 16, §III with f = log sum_k
// exp(w_k.x) - w_y.x), bf16 features, one pass over X, whole rows per CTA pair.
//
// For K this small both contractions of the gradient are thin:
//   Z = X_tile W^T           (16 rows x 16 classes, summed over d)
//   G += X_tile^T R          (d features x 16 classes, summed over the rows)
// and the step is bound by reading X once.  A cluster of two CTAs (one per
// SM) streams 16-row tiles; CTA r holds the tile's features
// [r ld/2, (r + 1) ld/2) (16 x ld/2 bf16, laid out as 64-feature blocks of 16
// rows with 128-byte swizzle by 3-D TMA copies of box_blocks blocks each) in a
// ring of slots, so four 48 KB slots are in flight at d = 3072:
//   1. eight warps form the partial logits of the CTA's features with
//      warp-level mma.sync (m16n8k16, bf16 in, fp32 out), each over a
//      sixteenth of d, with its slice of W^T held in registers for the whole
//      step, and hand them over through shared memory;
//   2. two warps of their own (even and odd tiles) sum them, send the CTA's
//      16 x 16 block to the other CTA with st.async into distributed shared
//      memory, add the two blocks in rank order (so both CTAs form the same
//      R) and form R = softmax(Z) - onehot(y) (zero past K and past the
//      partition's rows) in bf16, in the no-swizzle K-major operand layout.
//      The rounding uses error feedback: each entry's rounding error is
//      added to the same entry (row position, class) of the warp's next tile
//      of the run before that one is rounded, so over a run the errors
//      telescope instead of adding up.  Rounded independently, entries of
//      rows with alike softmax values round alike, and with non-negative
//      features those errors add up coherently over the rows of R^T X;
//   3. the same eight warps copy the half tile, transposed, into tensor memory
//      (one lane per feature, two rows per 32-bit column: the K-major A
//      operand of the gradient MMA) and release the slot, so a slot is held
//      only for its load, the logits and the copy, not for the exchange of
//      step 2; kNA copies (and R blocks) rotate;
//   4. two threads, each for half of the 128-feature slices, issue
//      tcgen05.mma (M = 128 features, N = 16 classes, K = the 16 rows; A =
//      the tile's copy in tensor memory, B = the R block) into a TMEM
//      accumulator of the CTA's half of G^T that spans the pair's run of
//      tiles in a partition; their two commits free the copy and the R block.
// No data leaves the pair before the end of a run; then the eight warps write
// the run's G^T halves into one partial (one item per pair and partition).
// With the fused tail the same grid then commits and decodes: after a grid
// barrier each CTA sums, for its slice of the columns, every partition's items
// in item order, scales by 1/m_e and writes the stores, then (after a CTA
// barrier) decodes and updates the same columns with the coefficients it
// derived from the mask; otherwise separate commit and decode kernels follow.
// Every wait is bounded; the TMEM allocation is released on every path.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstring>

#include "rows_tail.cuh"
#include "tc_common.cuh"

namespace pgc {

namespace {

constexpr int kRR = kRowsTileRows;       // rows per tile
static_assert(kRR == 16, "16-row tiles (mma.sync M = 16, tcgen05 K = 16)");
constexpr uint32_t kBlk = kRR * 128;      // one 64-feature block of the tile
constexpr int kPairCtas = 2;             // CTAs per cluster: feature halves
constexpr int kFw = 8;                   // forward warps (warps 2..9)
constexpr int kRWarp = 2 + kFw;          // the residual warps (even and odd tiles)
constexpr int kNRes = 2;
constexpr int kMWarp2 = kRWarp + kNRes;  // the second MMA-issuing warp (warp 1 is the first)
constexpr int kRThreads = 64 + 32 * kFw + 32 * kNRes + 32;
// 16-feature steps per forward warp at the largest ld
constexpr int kMaxKs = (int)(kRowsMaxLd / kPairCtas / (16 * kFw));
constexpr uint32_t kZp = kRR * 16 * 4;   // a 16 x 16 fp32 block of partial logits
constexpr uint32_t kRb = 16 * 16 * 2;    // R block (16 rows x 16 classes bf16)
constexpr int kNA = 3;                   // tiles whose gradient MMA may be pending (TMEM copies, R blocks)
constexpr int kTmemCols = 512;           // G^T half, then the kNA copies of a tile
constexpr uint32_t kAccCols = 192;       // G^T half: ld / 256 slices of 16 columns at the largest ld
constexpr uint32_t kAStride = 96;        // a copy: ld / 256 slices of 8 columns (16 rows of bf16)
static_assert(kRowsMaxLd / kPairCtas / 128 * 16 <= (int)kAccCols, "G^T half fits its columns");
static_assert(kRowsMaxLd / kPairCtas / 128 * 8 <= (int)kAStride, "a tile copy fits its columns");
static_assert(kAccCols + kNA * kAStride <= (uint32_t)kTmemCols, "tensor memory holds G^T and the copies");

__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo, uint32_t layout) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)layout << 61;
  return d;
}
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* tm, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
          smem_u32(dst)),
      "l"(tm), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a0, uint32_t& a1, uint32_t& a2, uint32_t& a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t& a0, uint32_t& a1, uint32_t& a2, uint32_t& a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
               : "r"(addr));
}
// 16 lanes x 8 columns from the warp: thread t writes lanes t/4 and t/4 + 8,
// columns 2 (t % 4) and 2 (t % 4) + 1 (the layout of an mma.sync accumulator)
__device__ __forceinline__ void tmem_st_16x256b(uint32_t taddr, uint32_t r0, uint32_t r1, uint32_t r2, uint32_t r3) {
  asm volatile("tcgen05.st.sync.aligned.16x256b.x1.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr), "r"(r0), "r"(r1), "r"(r2),
               "r"(r3)
               : "memory");
}
// K position of tile row r in the gradient MMA: the tensor-memory copy puts
// row pair p (rows 2p, 2p + 1) in column 2p (p < 4) or 2 (p - 4) + 1, so R
// is laid out with the same order of its K rows
__device__ __forceinline__ int k_of_row(int r) {
  const int p = r >> 1;
  return 2 * (p < 4 ? 2 * p : 2 * p - 7) + (r & 1);
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// D (+)= A B with A in tensor memory (K-major, one row per lane), B in shared memory
__device__ __forceinline__ void umma_ta_fresh(uint32_t tmem_d, uint32_t tmem_a, uint64_t db, uint32_t idesc) {
  asm volatile("tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, 0;" ::"r"(tmem_d), "r"(tmem_a), "l"(db),
               "r"(idesc)
               : "memory");
}
__device__ __forceinline__ void umma_ta_acc(uint32_t tmem_d, uint32_t tmem_a, uint64_t db, uint32_t idesc) {
  asm volatile("tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, 1;" ::"r"(tmem_d), "r"(tmem_a), "l"(db),
               "r"(idesc)
               : "memory");
}
// shared::cta address -> the same offset in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t mapa_u32(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_async_v4(uint32_t raddr, float4 v, uint32_t rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                   raddr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rbar)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive_remote(uint32_t rbar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(rbar) : "memory");
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
// bounded wait with cluster-scope acquire (the data came from the other CTA)
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
// Element (class k, tile row r) of the R block in the K-major layout without
// swizzle: 8 x 8 core matrices (8 classes x 16 bytes of rows), the core of
// row chunk r/8 and class group k/8 at (r/8)*256 + (k/8)*128.
__device__ __forceinline__ uint32_t r_offset(int k, int r) {
  return (uint32_t)((r >> 3) * 256 + (k >> 3) * 128 + (k & 7) * 16 + (r & 7) * 2);
}
}  // namespace

// Shared memory of a CTA: slots of its half tile, two sets (tile parity) of
// the forward warps' partial logits (the fused tail's decode plan reuses
// them), two blocks for the other CTA's partial, kNA R blocks, barriers.
struct RowsSmem {
  uint32_t slot_bytes, zpart, zpeer, rblk, bars, total;
};
constexpr int kRowsBars = 2 * kRowsMaxSlots + 3 * kNA + 8 + 4;
__host__ __device__ static RowsSmem rows_smem(int64_t ld, int nslots) {
  RowsSmem s;
  s.slot_bytes = (uint32_t)(kRR * (ld / kPairCtas) * 2);
  s.zpart = (uint32_t)nslots * s.slot_bytes;
  s.zpeer = s.zpart + 2 * kFw * kZp;
  s.rblk = s.zpeer + 2 * kZp;
  s.bars = s.rblk + (uint32_t)kNA * kRb;
  s.total = s.bars + kRowsBars * 8 + 16;
  return s;
}
static_assert(2 * kFw * kZp >= sizeof(DecodePlan), "the decode plan fits the partial-logit area");

__global__ void __launch_bounds__(kRThreads, 1)
softmax_rows_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ RowsArgs a) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ int bar_flag;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = a.nslots;
  const RowsSmem L = rows_smem(a.ld, S);
  float* zpart = reinterpret_cast<float*>(sm + L.zpart);   // [2][kFw][16][16]
  float* zpeer = reinterpret_cast<float*>(sm + L.zpeer);   // [2][16][16] from the other CTA
  DecodePlan& plan = *reinterpret_cast<DecodePlan*>(zpart);  // the tail's, after the tiles
  uint8_t* rblk = sm + L.rblk;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L.bars);
  uint64_t* full = bars;                          // [S] half tile landed
  uint64_t* empty = bars + kRowsMaxSlots;         // [S] the forward warps are done with the half tile
  uint64_t* rready = bars + 2 * kRowsMaxSlots;    // [kNA] R block written
  uint64_t* a_full = rready + kNA;                // [kNA] the tile's copy in tensor memory written
  uint64_t* a_empty = a_full + kNA;               // [kNA] the tile's MMAs are done (copy, R block free)
  uint64_t* zready = a_empty + kNA;               // [2] every forward warp's partial written
  uint64_t* zfree = zready + 2;                   // [2] the residual warp has read them
  uint64_t* zpeer_full = zready + 4;              // [2] the other CTA's block arrived
  uint64_t* zpeer_empty = zready + 6;             // [2] the other CTA has read this CTA's block
  uint64_t* acc_full = zready + 8;
  uint64_t* acc_empty = acc_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 2);
  int* cta_err = reinterpret_cast<int*>(acc_full + 3);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = (int)cluster_rank();
  const int64_t ldh = a.ld / kPairCtas;          // features of this CTA
  const int nmt = (int)(ldh / 128);              // 128-feature M slices of the backward
  // this pair's tiles (split on the host)
  const int pair = (int)blockIdx.x / kPairCtas;
  const int t0 = a.pair_t0[pair], t1 = a.pair_t0[pair + 1];
  const int n = t1 - t0;

  if (threadIdx.x == 0) {
    *cta_err = 0;
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kFw);
    }
    for (int b = 0; b < kNA; ++b) {
      mbar_init(&rready[b], 1);
      mbar_init(&a_full[b], kFw);
      mbar_init(&a_empty[b], 2);         // the commits of both MMA issuers
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&zready[b], kFw);
      mbar_init(&zfree[b], 1);
      mbar_init(&zpeer_full[b], 1);
      mbar_init(&zpeer_empty[b], 1);
    }
    mbar_init(acc_full, 2);
    mbar_init(acc_empty, kFw);
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"((uint32_t)kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();
  // the other CTA's first two blocks may arrive before this CTA reaches them
  if (threadIdx.x == 0)
    for (int b = 0; b < 2 && b < n; ++b) mbar_arrive_expect_tx(&zpeer_full[b], kZp);
  tc_fence_before();
  cluster_sync_all();                    // both CTAs' barriers exist before any st.async
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (threadIdx.x == 0) grid_dep_launch();

  if (warp == 0 && lane == 0) {
    // ---- producer: this CTA's half of each tile ------------------------------
    bool ok = true;
    int issued = 0;
    const uint32_t bytes = L.slot_bytes;
    const int nkb = (int)(ldh / 64), kb0 = rank * nkb;
    // X does not change between steps: no wait for the previous kernel
    for (int i = 0; i < n && ok; ++i) {
      const int s = i % S;
      if (i >= S && !mbar_wait(&empty[s], ((i / S) - 1) & 1, a.status)) { ok = false; break; }
      mbar_arrive_expect_tx(&full[s], bytes);
      const int row0 = a.tiles[t0 + i].x;
      for (int z = 0; z < nkb; z += a.box_blocks)
        tma_load_3d(sm + (size_t)s * bytes + (size_t)z * kBlk, &tmX, 0, row0, kb0 + z, &full[s]);
      ++issued;
    }
    if (!ok) atomicExch(cta_err, 1);
    for (int s = 0; s < S && s < issued; ++s) {
      const int last = ((issued - 1 - s) / S) * S + s;
      mbar_wait(&full[s], (last / S) & 1, a.status);
    }
  } else if ((warp == 1 || warp == kMWarp2) && lane == 0) {
    // ---- backward MMAs: G^T[f][k] += sum_r X[r][f] R[r][k] ------------------
    // Two issuing threads, each with half of the 128-feature slices (they
    // write different accumulator columns): a single thread issues these
    // small MMAs more slowly than the tiles arrive.  Each commits its own
    // MMAs; the barriers they free count both.
    constexpr uint32_t id_bwd = idesc_bf16_f32(128, 16, false, false);
    const int mt0 = warp == 1 ? 0 : (nmt + 1) / 2, mt1 = warp == 1 ? (nmt + 1) / 2 : nmt;
    bool ok = true;
    int run = 0;
    for (int i = 0; i < n && ok; ++i) {
      const int ab = i % kNA;
      const int4 tl = a.tiles[t0 + i];
      const bool first = (tl.w & 1) || i == 0, last = (tl.w & 2) || i == n - 1;
      if (!mbar_wait(&a_full[ab], (i / kNA) & 1, a.status) || !mbar_wait(&rready[ab], (i / kNA) & 1, a.status)) {
        ok = false;
        break;
      }
      if (first && run > 0 && !mbar_wait(acc_empty, (run - 1) & 1, a.status)) { ok = false; break; }
      tc_fence_after();
      const uint64_t db = sdesc(smem_u32(rblk + ab * kRb), 256, 128, 0);
      // slice mt: its 128 features x 16 rows are columns kAccCols + ab kAStride + 8 mt ..
      const uint32_t ta = tmem + kAccCols + (uint32_t)ab * kAStride;
      for (int mt = mt0; mt < mt1; ++mt) {
        const uint32_t d = tmem + (uint32_t)(mt * 16), am = ta + (uint32_t)(mt * 8);
        if (first) umma_ta_fresh(d, am, db, id_bwd);
        else umma_ta_acc(d, am, db, id_bwd);
      }
      umma_commit(&a_empty[ab]);
      if (last) {
        umma_commit(acc_full);
        ++run;
      }
    }
    if (!ok) atomicExch(cta_err, 1);
  } else if (warp >= kRWarp && warp < kRWarp + kNRes) {
    // ---- residual: the pair's logits, R = softmax(Z) - onehot(y) ------------
    // Two warps, for the even and the odd tiles (every buffer and barrier of
    // the exchange is per tile parity), so one tile's exchange with the other
    // CTA overlaps the next tile's.  lane: row lane / 2, classes 8 (lane & 1)
    // .. + 7.  The R block i % kNA is written once tile i - kNA's MMAs have
    // read it (a_empty).  ef: the rounding errors of this lane's entries in
    // the warp's previous tile of the same run (error feedback).
    const int r = lane >> 1, kh = (lane & 1) * 8;
    const uint32_t peer = (uint32_t)(rank ^ 1);
    bool ok = true;
    float ef[8];
    int ef_item = -1;
    for (int i = warp - kRWarp; i < n && ok; i += kNRes) {
      const int b = i & 1;
      const int4 tl = a.tiles[t0 + i];
      const bool valid = r < tl.y;
      if (tl.z != ef_item) {                             // a new run: nothing carried in
        ef_item = tl.z;
#pragma unroll
        for (int c = 0; c < 8; ++c) ef[c] = 0.f;
      }
      const int lab = valid ? a.y[tl.x + r] : -1;        // fetched before the waits
      if (!__all_sync(0xffffffffu, mbar_wait(&zready[b], (i >> 1) & 1, a.status))) { ok = false; break; }
      float z[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) z[c] = 0.f;
      const float* zs = zpart + (size_t)b * kFw * (kRR * 16) + r * 16 + kh;
#pragma unroll
      for (int w = 0; w < kFw; ++w) {
        const float4 u0 = *reinterpret_cast<const float4*>(zs + w * (kRR * 16));
        const float4 u1 = *reinterpret_cast<const float4*>(zs + w * (kRR * 16) + 4);
        z[0] += u0.x; z[1] += u0.y; z[2] += u0.z; z[3] += u0.w;
        z[4] += u1.x; z[5] += u1.y; z[6] += u1.z; z[7] += u1.w;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&zfree[b]);             // the forward warps may refill zpart[b]
      // this CTA's block to the other CTA, once it has read the one sent two tiles ago
      if (i >= 2 && !__all_sync(0xffffffffu, wait_cluster(&zpeer_empty[b], ((i >> 1) - 1) & 1, a.status))) {
        ok = false;
        break;
      }
      {
        const uint32_t dst = mapa_u32(smem_u32(zpeer + (size_t)b * (kRR * 16) + r * 16 + kh), peer);
        const uint32_t rbar = mapa_u32(smem_u32(&zpeer_full[b]), peer);
        st_async_v4(dst, make_float4(z[0], z[1], z[2], z[3]), rbar);
        st_async_v4(dst + 16, make_float4(z[4], z[5], z[6], z[7]), rbar);
      }
      if (!__all_sync(0xffffffffu, wait_cluster(&zpeer_full[b], (i >> 1) & 1, a.status))) { ok = false; break; }
      const float* zp = zpeer + (size_t)b * (kRR * 16) + r * 16 + kh;
      float y[8];
      {
        const float4 u0 = *reinterpret_cast<const float4*>(zp);
        const float4 u1 = *reinterpret_cast<const float4*>(zp + 4);
        y[0] = u0.x; y[1] = u0.y; y[2] = u0.z; y[3] = u0.w; y[4] = u1.x; y[5] = u1.y; y[6] = u1.z; y[7] = u1.w;
      }
      __syncwarp();
      if (i + 2 < n) {
        if (lane == 0) {
          mbar_arrive_expect_tx(&zpeer_full[b], kZp);     // the other CTA's block of tile i + 2
          mbar_arrive_remote(mapa_u32(smem_u32(&zpeer_empty[b]), peer));
        }
      }
      // the same sum in both CTAs: rank 0's block first
#pragma unroll
      for (int c = 0; c < 8; ++c) z[c] = rank == 0 ? z[c] + y[c] : y[c] + z[c];
      float m = -INFINITY;
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (kh + c < a.K) m = fmaxf(m, z[c]);
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
      float e[8], sum = 0.f;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        e[c] = kh + c < a.K ? expf(z[c] - m) : 0.f;
        sum += e[c];
      }
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      const float inv = 1.0f / sum;
      if (i >= kNA && !__all_sync(0xffffffffu, mbar_wait(&a_empty[i % kNA], ((i / kNA) - 1) & 1, a.status))) {
        ok = false;
        break;
      }
      uint8_t* blk = rblk + (i % kNA) * kRb;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        const int k = kh + c;
        __nv_bfloat16 q = __float2bfloat16_rn(0.f);
        if (valid && k < a.K) {
          const float v = e[c] * inv - (k == lab ? 1.f : 0.f) + ef[c];
          q = __float2bfloat16_rn(v);
          ef[c] = v - __bfloat162float(q);
        }
        *reinterpret_cast<__nv_bfloat16*>(blk + r_offset(k, k_of_row(r))) = q;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&rready[i % kNA]);
    }
    if (!ok) atomicExch(cta_err, 1);
  } else if (warp >= 2 && warp < kRWarp) {
    // ---- forward (8 warps), run drain (all 8) ---------------------------------
    const int fw = warp - 2;
    const int nks = (int)(ldh / (16 * kFw));    // 16-feature steps of this warp
    const int f0 = fw * nks * 16;               // first feature of this warp within the half
    const int g = lane >> 2, tq = lane & 3;
    grid_dep_wait();                            // W is the previous step's update
    // B fragments of W^T for this warp's features: b0 = W[n][k0 + 2tq ..],
    // b1 = W[n][k0 + 8 + 2tq ..], n = 8 nb + g
    uint32_t wf[kMaxKs][2][2];
#pragma unroll
    for (int ks = 0; ks < kMaxKs; ++ks)
#pragma unroll
      for (int nb = 0; nb < 2; ++nb) {
        wf[ks][nb][0] = wf[ks][nb][1] = 0u;
        if (ks < nks) {
          const uint16_t* wr = a.wb + (int64_t)(8 * nb + g) * a.ld + rank * ldh + f0 + ks * 16 + 2 * tq;
          wf[ks][nb][0] = *reinterpret_cast<const uint32_t*>(wr);
          wf[ks][nb][1] = *reinterpret_cast<const uint32_t*>(wr + 8);
        }
      }
    // ldmatrix row of this lane: matrix m = lane / 8 (rows 8 (m & 1) .., features 8 (m >> 1) ..)
    const int lr = ((lane >> 3) & 1) * 8 + (lane & 7), lk = (lane >> 4) * 8;
    // The half tile j, transposed, into tensor memory as the gradient MMA's A
    // operand: this warp writes lane quarter q (features 32 q .. of each
    // 128-feature slice) of the slices of parity h; then slot j % S is
    // released.  The copy of tile j - kNA must have been read by its MMAs.
    // ldmatrix.trans of four 8 x 8 blocks (rows 0-7 / 8-15 x features fb ..
    // fb + 7 / fb + 8 .. fb + 15) gives thread t rows 2 (t % 4), 2 (t % 4) + 1
    // of each row half of features t / 4 and 8 + t / 4 (row pairs t % 4 and
    // 4 + t % 4), stored as columns 2 (t % 4) and 2 (t % 4) + 1 of lanes t / 4
    // and t / 4 + 8 (k_of_row gives R the same order of its K rows).
    auto copy_tile = [&](int j) -> bool {
      if (j >= kNA && !__all_sync(0xffffffffu, mbar_wait(&a_empty[j % kNA], ((j / kNA) - 1) & 1, a.status)))
        return false;
      tc_fence_after();
      const int q = warp & 3, h = (warp - 2) >> 2;
      const uint32_t xj = smem_u32(sm + (size_t)(j % S) * L.slot_bytes);
      const uint32_t ta = tmem + ((uint32_t)(q * 32) << 16) + kAccCols + (uint32_t)(j % kNA) * kAStride;
      const int mi = lane >> 3, mr = ((mi & 1) << 3) + (lane & 7);
      for (int mt = h; mt < nmt; mt += 2) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int f = mt * 128 + q * 32 + hh * 16 + ((mi >> 1) << 3);
          const uint32_t ad = xj + (uint32_t)((f >> 6) * kBlk + mr * 128 + ((((f & 63) >> 3) ^ (mr & 7)) << 4));
          uint32_t v0, v1, v2, v3;
          ldsm_x4_trans(ad, v0, v1, v2, v3);
          tmem_st_16x256b(ta + ((uint32_t)(hh * 16) << 16) + (uint32_t)(mt * 8), v0, v1, v2, v3);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&a_full[j % kNA]);
        mbar_arrive(&empty[j % S]);
      }
      return true;
    };
    bool ok = true;
    int run = 0;
    int pending = -1;
    for (int i = 0; i < n; ++i) {
      const int s = i % S, b = i & 1;
      const int4 tl = a.tiles[t0 + i];
      const bool last = (tl.w & 2) || i == n - 1;
      if (!__all_sync(0xffffffffu, mbar_wait(&full[s], (i / S) & 1, a.status))) { ok = false; break; }
      const uint32_t xs = smem_u32(sm + (size_t)s * L.slot_bytes);
      // four independent accumulator chains (class halves x even / odd steps)
      float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
      float d0[4] = {0.f, 0.f, 0.f, 0.f}, d1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ks = 0; ks < kMaxKs; ++ks) {
        if (ks < nks) {
          const int f = f0 + ks * 16 + lk;
          const uint32_t ad = xs + (uint32_t)((f >> 6) * kBlk + lr * 128 + ((((f & 63) >> 3) ^ (lr & 7)) << 4));
          uint32_t a0, a1, a2, a3;
          ldsm_x4(ad, a0, a1, a2, a3);
          if (ks & 1) {
            mma16816(d0, a0, a1, a2, a3, wf[ks][0][0], wf[ks][0][1]);
            mma16816(d1, a0, a1, a2, a3, wf[ks][1][0], wf[ks][1][1]);
          } else {
            mma16816(c0, a0, a1, a2, a3, wf[ks][0][0], wf[ks][0][1]);
            mma16816(c1, a0, a1, a2, a3, wf[ks][1][0], wf[ks][1][1]);
          }
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        c0[j] += d0[j];
        c1[j] += d1[j];
      }
      // the residual warp has read this buffer's previous tile (i - 2)
      if (i >= 2 && !__all_sync(0xffffffffu, mbar_wait(&zfree[b], ((i >> 1) - 1) & 1, a.status))) {
        ok = false;
        break;
      }
      // partial logits: rows g, g + 8; classes 2tq, 2tq + 1 (+ 8 for c1)
      float* zp = zpart + (size_t)(b * kFw + fw) * (kRR * 16);
      *reinterpret_cast<float2*>(zp + g * 16 + 2 * tq) = make_float2(c0[0], c0[1]);
      *reinterpret_cast<float2*>(zp + g * 16 + 8 + 2 * tq) = make_float2(c1[0], c1[1]);
      *reinterpret_cast<float2*>(zp + (g + 8) * 16 + 2 * tq) = make_float2(c0[2], c0[3]);
      *reinterpret_cast<float2*>(zp + (g + 8) * 16 + 8 + 2 * tq) = make_float2(c1[2], c1[3]);
      __syncwarp();
      if (lane == 0) mbar_arrive(&zready[b]);
      // the previous tile's copy waits until this tile's logits are handed
      // over, so that the logits do not wait for tile i - kNA's MMAs; the last
      // tile of a run is copied at once (its drain needs its MMAs)
      if (pending >= 0) {
        if (!copy_tile(pending)) { ok = false; break; }
        pending = -1;
      }
      if (!last) {
        pending = i;
      } else if (!copy_tile(i)) {
        ok = false;
        break;
      }
      if (last) {
        // end of the pair's run in a partition: this CTA's G^T slices -> its
        // half of the run's partial
        if (!__all_sync(0xffffffffu, mbar_wait(acc_full, run & 1, a.status))) { ok = false; break; }
        // warps w and w + 4 share TMEM lane quarter w % 4 and split the
        // slices: pairs (2j, 2j + 1) go to the first, then the second, ...
        tc_fence_after();
        const int q = warp & 3, half = (warp - 2) >> 2;
        float* dst = a.partials + (int64_t)tl.z * a.P + rank * ldh;
        for (int mt = 2 * half; mt < nmt; mt += 4) {
          uint32_t gv[32];
          tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(mt * 16), gv);   // slices mt, mt + 1
          tmem_ld_wait();
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (mt + h < nmt) {
              const int f = (mt + h) * 128 + q * 32 + lane;
#pragma unroll
              for (int k = 0; k < 16; ++k)
                if (k < a.K) dst[(int64_t)k * a.ld + f] = __uint_as_float(gv[16 * h + k]);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty);
      }
      if (last) ++run;
    }
    if (!ok) atomicExch(cta_err, 1);
  }
  __syncthreads();
  tc_fence_before();
  cluster_sync_all();                    // no st.async or remote arrive is still aimed at this CTA
  tc_fence_after();
  if (a.tail && !*cta_err) {
    // ---- fused tail: commit, then decode + SGD (rows_tail.cuh); the decode
    // plan goes where the partial logits were, the committed gradients of
    // the short route where the slots were
    rows_fused_tail(a, *reinterpret_cast<DecodePlan*>(zpart), sm, (int64_t)S * L.slot_bytes, &bar_flag);
  }
  if (warp == 1) {
    // after a failure, wait (bounded) for the last commit before releasing TMEM
    if (*cta_err && lane == 0 && n > 0) mbar_wait(&a_empty[(n - 1) % kNA], ((n - 1) / kNA) & 1, a.status);
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)kTmemCols)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int rows_slots(int64_t ld) {
  if (ld % (128 * kPairCtas) != 0 || ld > kRowsMaxLd) return 0;
  int s = kRowsMaxSlots;
  while (s >= 2 && rows_smem(ld, s).total + 1024 > kRowsSmemBudget) --s;
  return s >= 2 ? s : 0;
}

int rows_box_blocks(int64_t ld, int requested) {
  const int nkb = (int)(ld / kPairCtas / 64);   // blocks of one CTA's half
  if (nkb < 1) return 0;
  if (requested >= 1 && nkb % requested == 0) return requested;
  for (int b = 8; b >= 1; --b)
    if (nkb % b == 0) return b;
  return 1;
}

static size_t rows_smem_bytes(int64_t ld, int nslots) { return 1024 + rows_smem(ld, nslots).total; }

static cudaLaunchConfig_t rows_config(int64_t ld, int nslots, int nctas, cudaLaunchAttribute* attr, bool pdl,
                                      cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)nctas);
  cfg.blockDim = dim3(kRThreads);
  cfg.dynamicSmemBytes = rows_smem_bytes(ld, nslots);
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kPairCtas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cfg;
}

int rows_max_ctas(int64_t ld, int nslots) {
  const size_t smem = rows_smem_bytes(ld, nslots);
  if (cudaFuncSetAttribute(softmax_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess)
    return 0;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = rows_config(ld, nslots, kPairCtas, attr, false, 0);
  int nc = 0;
  if (cudaOccupancyMaxActiveClusters(&nc, softmax_rows_kernel, &cfg) != cudaSuccess) return 0;
  return nc * kPairCtas;   // every pair co-resident (the fused tail's grid barriers need it)
}

cudaError_t launch_softmax_rows(const void* tmX, const RowsArgs& a, int nctas, cudaStream_t st) {
  if (a.ntiles <= 0) return cudaSuccess;
  if (nctas < kPairCtas || nctas % kPairCtas != 0 || a.nslots < 2 || a.nslots > kRowsMaxSlots)
    return cudaErrorInvalidValue;
  if (a.box_blocks < 1 || (a.ld / kPairCtas / 64) % a.box_blocks != 0) return cudaErrorInvalidValue;
  const size_t smem = rows_smem_bytes(a.ld, a.nslots);
  cudaError_t e = cudaFuncSetAttribute(softmax_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = rows_config(a.ld, a.nslots, nctas, attr, a.pdl != 0, st);
  CUtensorMap x;
  std::memcpy(&x, tmX, sizeof(CUtensorMap));
  return cudaLaunchKernelEx(&cfg, softmax_rows_kernel, x, a);
}

}  // namespace pgc
