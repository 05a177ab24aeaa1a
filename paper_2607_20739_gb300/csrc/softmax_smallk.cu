// Softmax gradient for few classes (K <= 16, §III with f = log sum_k
// exp(w_k.x) - w_y.x), bf16 features, one pass over X.
//
// For K this small the two contractions of the gradient,
//   Z = X_tile W^T            (128 rows x 16 classes, summed over d)
//   G += X_tile^T R           (d features x 16 classes, summed over rows)
// are thin, and the work is bound by reading X.  The kernel reads every X
// tile from HBM exactly once: a cluster of 8 CTAs splits the feature axis, each
// CTA keeping its slice of the tile (128 rows x d/8 features) in shared memory
// for both contractions.  Per tile:
//   1. each CTA computes its partial Z over its feature slice (tcgen05.mma,
//      M = 128 rows, N = 16 classes, accumulator in TMEM);
//   2. the partial Z rows are sent to their owner CTA (rank = row / 16) with
//      st.async into distributed shared memory; the owner sums the 8 slices,
//      forms R = softmax(Z) - onehot(y) for its 16 rows and sends it to all 8
//      CTAs with bulk copies (cp.async.bulk shared::cluster) as two bf16
//      blocks, R_hi = bf16(R) and R_lo = bf16(R - R_hi): bf16 alone is not
//      enough when the rows' softmax values are alike, since their rounding
//      errors then add up coherently over the rows of the contraction;
//   3. each CTA accumulates its slice of G^T (M = 128 features, N = 16
//      classes, K = the tile's rows; B = R_hi, then B = R_lo) in TMEM,
//      reading the same resident X slice, now as an MN-major operand.
// When a cluster's run of tiles leaves a partition its G^T slices are written
// as one partial (one item per cluster and partition); a separate commit
// kernel sums the items of each partition, scales by 1/m_e and writes the
// stores.  Every wait is bounded.
//
// Cross-CTA protocol (single zred buffer, double-buffered R and X slots):
//   CTA p sends its Z(i) rows only after every owner's R(i-1) block arrived in
//   p (so every owner has finished reading zred for tile i-1); an owner sends
//   R(i+2) into p's R buffer only after p's Z(i+2) arrived, which p sends after
//   its MMAs of tile i (the previous user of that R buffer) completed.
#include <cuda.h>

#include <cstring>

#include "tail.cuh"

namespace pgc {

namespace {

constexpr int kCS = 8;                 // CTAs per cluster (feature slices)
constexpr int kRows = kSmallKRows;     // rows per tile (MMA M of the forward)
static_assert(kRows == 128, "the forward accumulator layout assumes M = 128");
constexpr int kTileCache = 128;        // tile descriptors kept in shared memory
constexpr int kNC = 16;                // padded classes (MMA N)
constexpr int kThreads = 192;          // producer, MMA, 4 epilogue warps
constexpr uint32_t kBox = kRows * 64 * 2;      // one 128 x 64 bf16 X box
constexpr uint32_t kWBox = kNC * 64 * 2;       // one 16 x 64 bf16 W box
constexpr uint32_t kZPart = 16 * kNC * 4;      // 16 rows of partial Z: one source's share
constexpr uint32_t kRBlock = 16 * kNC * 2;     // 16 rows of R (bf16)
constexpr uint32_t kTmemCols = 128;

__device__ __forceinline__ uint32_t cl_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cl_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cl_count() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cl_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// shared::cta address -> the same offset in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t mapa(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_async_v4(uint32_t raddr, float4 v, uint32_t rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                   raddr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rbar)
               : "memory");
}
__device__ __forceinline__ void bulk_s2cluster(uint32_t rdst, const void* src, uint32_t bytes, uint32_t rbar) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   rdst),
               "r"(smem_u32(src)), "r"(bytes), "r"(rbar)
               : "memory");
}
// wait with cluster-scope acquire (the data came from other CTAs' st.async)
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
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
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, int* status) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 0; it < kWaitMaxIters; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 63u) == 63u && globaltimer_ns() - t0 > kWaitMaxNs) break;
  }
  atomicOr(status, kErrWaitTimeout);
  return false;
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* tm, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(dst)),
      "l"(tm), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// tcgen05 shared-memory descriptor: start, leading / stride byte offsets (16-byte
// units), version 1, layout (0: no swizzle, 2: 128-byte swizzle).
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo, uint32_t layout) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)layout << 61;
  return d;
}
// kind::f16 instruction descriptor: fp32 accumulate, bf16 A and B.
__host__ __device__ constexpr uint32_t idesc(int M, int N, bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(id), "r"(acc)
      : "memory");
}
// accumulate into D (no predicate computation on the issue path)
__device__ __forceinline__ void mma_acc(uint32_t d, uint64_t a, uint64_t b, uint32_t id) {
  asm volatile("tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, 1;" ::"r"(d), "l"(a), "l"(b), "r"(id) : "memory");
}
__device__ __forceinline__ void commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int k = 0; k < 16; ++k) v[k] = __uint_as_float(r[k]);
}
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Element (class k, tile row r) of the R tile, in the K-major layout without
// swizzle: 8 x 8 core matrices (8 classes x 16 bytes of rows), the core of
// row chunk r/8 and class group k/8 at (r/8)*256 + (k/8)*128.
__device__ __forceinline__ uint32_t r_offset(int k, int r) {
  return (uint32_t)((r >> 3) * 256 + (k >> 3) * 128 + (k & 7) * 16 + (r & 7) * 2);
}

}  // namespace

// Shared-memory plan; offsets from the 1024-byte aligned base.
struct SkSmem {
  uint32_t slots, slot_bytes, wsm, zred, rstage, rbuf, rbuf_lo, tiles, bars, total;
};
__host__ __device__ static SkSmem sk_smem(int nper) {
  SkSmem s;
  const int even = (nper + 1) & ~1;
  s.slot_bytes = (uint32_t)even * kBox;
  s.slots = 0;
  s.wsm = 2 * s.slot_bytes;
  s.zred = s.wsm + (uint32_t)((nper * kWBox + 1023) & ~1023);
  s.rstage = s.zred + kCS * kZPart;
  s.rbuf = s.rstage + 4 * kRBlock;          // staging: [slot][hi, lo]
  s.rbuf_lo = s.rbuf + 2 * kCS * kRBlock;
  s.tiles = s.rbuf_lo + 2 * kCS * kRBlock;
  s.bars = s.tiles + kTileCache * 16;
  s.total = s.bars + 32 * 8 + 16;
  return s;
}

__global__ void __launch_bounds__(kThreads, 1)
softmax_smallk_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW, SmallKArgs a) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SkSmem L = sk_smem(a.nper);
  uint8_t* slot0 = sm + L.slots;
  uint8_t* wsm = sm + L.wsm;
  float* zred = reinterpret_cast<float*>(sm + L.zred);
  uint8_t* rstage = sm + L.rstage;
  uint8_t* rbuf = sm + L.rbuf;
  uint8_t* rbuf_lo = sm + L.rbuf_lo;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L.bars);
  uint64_t* slot_full = bars + 0;    // [2]
  uint64_t* slot_empty = bars + 2;   // [2]
  uint64_t* wfull = bars + 4;
  uint64_t* zacc_full = bars + 5;    // [2]
  uint64_t* zacc_empty = bars + 7;   // [2]
  uint64_t* zred_full = bars + 9;
  uint64_t* rfull = bars + 10;       // [2]
  uint64_t* gfull = bars + 12;       // [2]
  uint64_t* gempty = bars + 14;      // [2]
  uint64_t* mma_done = bars + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);
  int4* tcache = reinterpret_cast<int4*>(sm + L.tiles);  // this cluster's first tile descriptors
  __shared__ int cta_err;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cl_rank();
  const int kb0 = (int)rank * a.nper;
  const int nk = max(0, min(a.nkb - kb0, a.nper));       // k blocks (64 features) of this slice
  const int nmt = (nk + 1) / 2;                           // 128-feature M tiles of the backward

  // tiles of this cluster
  const int64_t ncl = cl_count(), cid = cl_id();
  const int t0 = (int)((int64_t)a.ntiles * cid / ncl), t1 = (int)((int64_t)a.ntiles * (cid + 1) / ncl);
  const int n = t1 - t0;

  for (int i = threadIdx.x; i < n && i < kTileCache; i += blockDim.x) tcache[i] = a.tiles[t0 + i];
  auto tile_desc = [&](int i) { return i < kTileCache ? tcache[i] : a.tiles[t0 + i]; };
  if (threadIdx.x == 0) {
    cta_err = 0;
    for (int i = 0; i < 2; ++i) {
      mbar_init(&slot_full[i], 1);
      mbar_init(&slot_empty[i], 1);
      mbar_init(&zacc_full[i], 1);
      mbar_init(&zacc_empty[i], 4);
      mbar_init(&rfull[i], 1);
      mbar_init(&gfull[i], 1);
      mbar_init(&gempty[i], 4);
    }
    mbar_init(wfull, 1);
    mbar_init(zred_full, 1);
    mbar_init(mma_done, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();
  // the receive barriers expect their first tiles before any peer can send
  if (threadIdx.x == 64) {
    mbar_arrive_expect_tx(zred_full, kCS * kZPart);
    mbar_arrive_expect_tx(&rfull[0], 2 * kCS * kRBlock);
    mbar_arrive_expect_tx(&rfull[1], 2 * kCS * kRBlock);
  }
  fence_before();
  cl_sync();
  fence_after();
  const uint32_t tmem = *tmem_slot;
  // TMEM columns: partial Z [2][16] at 0, G^T [2][3 M tiles][16] at 32
  auto zacc_col = [](int s) { return (uint32_t)(s * kNC); };
  auto gacc_col = [](int g) { return (uint32_t)(2 * kNC + g * 3 * kNC); };
  if (threadIdx.x == 0) grid_dep_launch();

  if (warp == 0 && lane == 0) {
    // ---- producer: X slices of the tiles, W slice once ---------------------
    bool ok = true;
    int issued = 0;
    auto load_x = [&](int i) {
      const int s = i & 1;
      const int4 tl = tile_desc(i);
      mbar_arrive_expect_tx(&slot_full[s], (uint32_t)nk * kBox);
      for (int j = 0; j < nk; ++j)
        tma_load_2d(slot0 + s * L.slot_bytes + j * kBox, &tmX, (kb0 + j) * 64, tl.x, &slot_full[s]);
      ++issued;
    };
    // X does not change between steps: the first two tiles load while the
    // previous kernel finishes; W (updated by it) only after the wait
    for (int i = 0; i < n && i < 2; ++i) load_x(i);
    grid_dep_wait();
    mbar_arrive_expect_tx(wfull, (uint32_t)nk * kWBox);
    for (int j = 0; j < nk; ++j) tma_load_2d(wsm + j * kWBox, &tmW, (kb0 + j) * 64, 0, wfull);
    for (int i = 2; i < n; ++i) {
      if (!mbar_wait(&slot_empty[i & 1], ((i >> 1) - 1) & 1, a.status)) { ok = false; break; }
      load_x(i);
    }
    if (!ok) atomicExch(&cta_err, 1);
    // nothing may land after the CTA exits: wait for every slot's last fill
    for (int s = 0; s < 2 && s < issued; ++s) {
      const int last = ((issued - 1 - s) >> 1) * 2 + s;
      mbar_wait(&slot_full[s], (last >> 1) & 1, a.status);
    }
    mbar_wait(wfull, 0, a.status);
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer ----------------------------------------------------------
    // Forward of tile f once its X slice landed (at most two tiles ahead of
    // the backward: two X slots); backward of tile b as soon as its R block
    // arrived.  Whichever is ready goes first, so a slot is released as soon
    // as its exchange completes.  Readiness is probed with test_wait, which
    // never suspends the thread; descriptors are formed once per operand and
    // stepped by constants (the address field counts 16-byte units).
    constexpr uint32_t id_fwd = idesc(kRows, kNC, false, false);
    constexpr uint32_t id_bwd = idesc(kRows, kNC, true, false);
    bool ok = mbar_wait(wfull, 0, a.status);
    int seg = -1, f = 0, b = 0;
    uint64_t t_idle = 0;
    uint32_t spins = 0;
    while (ok && b < n) {
      bool did = false;
      if (b < f && mbar_test_wait(&rfull[b & 1], (b >> 1) & 1)) {
        const int s = b & 1;
        const int4 tl = tile_desc(b);
        const bool first = (tl.w & 1) || b == 0, last = (tl.w & 2) || b == n - 1;
        const int g = (seg + (first ? 1 : 0)) & 1;
        if (!first || seg + 1 < 2 || mbar_test_wait(&gempty[g], (((seg + 1) >> 1) - 1) & 1)) {
          if (first) ++seg;
          if (b + 2 < n) mbar_arrive_expect_tx(&rfull[s], 2 * kCS * kRBlock);
          fence_after();
          const uint32_t base = smem_u32(slot0 + s * L.slot_bytes);
          const uint64_t db = sdesc(smem_u32(rbuf + s * kCS * kRBlock), 256, 128, 0);
          const uint64_t dbl = sdesc(smem_u32(rbuf_lo + s * kCS * kRBlock), 256, 128, 0);
          for (int mt = 0; mt < nmt; ++mt) {
            const uint64_t da = sdesc(base + 2 * mt * kBox, kBox, 1024, 2);
            const uint32_t d = tmem + gacc_col(g) + mt * kNC;
            mma(d, da, db, id_bwd, first ? 0u : 1u);
#pragma unroll
            for (int kk = 1; kk < kRows / 16; ++kk) mma_acc(d, da + kk * 128, db + kk * 32, id_bwd);
#pragma unroll
            for (int kk = 0; kk < kRows / 16; ++kk) mma_acc(d, da + kk * 128, dbl + kk * 32, id_bwd);
          }
          commit(&slot_empty[s]);
          if (last) commit(&gfull[g]);
          ++b;
          did = true;
        }
      }
      if (!did && f < n && f - b < 2 && mbar_test_wait(&slot_full[f & 1], (f >> 1) & 1) &&
          (f < 2 || mbar_test_wait(&zacc_empty[f & 1], ((f >> 1) - 1) & 1))) {
        const int s = f & 1;
        fence_after();
        const uint64_t da0 = sdesc(smem_u32(slot0 + s * L.slot_bytes), 16, 1024, 2);
        const uint64_t db0 = sdesc(smem_u32(wsm), 16, 1024, 2);
        const uint32_t d = tmem + zacc_col(s);
        for (int j = 0; j < nk; ++j) {
          const uint64_t da = da0 + j * (kBox >> 4), db = db0 + j * (kWBox >> 4);
          mma(d, da, db, id_fwd, j != 0 ? 1u : 0u);
          mma_acc(d, da + 2, db + 2, id_fwd);
          mma_acc(d, da + 4, db + 4, id_fwd);
          mma_acc(d, da + 6, db + 6, id_fwd);
        }
        commit(&zacc_full[s]);
        ++f;
        did = true;
      }
      if (did) {
        t_idle = 0;
        spins = 0;
      } else {
        // bounded like every other wait: give up after kWaitMaxNs without progress
        if (t_idle == 0) t_idle = globaltimer_ns();
        if (++spins > kWaitMaxIters || ((spins & 63u) == 0 && globaltimer_ns() - t_idle > kWaitMaxNs)) {
          atomicOr(a.status, kErrWaitTimeout);
          ok = false;
        }
      }
    }
    if (!ok) atomicExch(&cta_err, 1);
  } else if (warp >= 2) {
    // ---- epilogue / reducer (128 threads) -----------------------------------
    const int t = threadIdx.x - 64;
    const int q = warp & 3;                       // TMEM lane quarter
    const int row = q * 32 + lane;                // tile row drained by this thread
    const int own = row >> 4;                     // owner CTA of that row
    const int j = t >> 3, cp = t & 7;             // reducer: my row j (of 16), classes 2cp, 2cp+1
    const uint32_t zred_remote = mapa(smem_u32(zred), (uint32_t)own) + rank * kZPart + (row & 15) * (kNC * 4);
    const uint32_t zbar_remote = mapa(smem_u32(zred_full), (uint32_t)own);
    bool ok = true;
    int seg = -1;
    bool waited = false;
    for (int i = 0; i < n && ok; ++i) {
      const int s = i & 1;
      const int4 tl = tile_desc(i);
      const bool first = (tl.w & 1) || i == 0, last = (tl.w & 2) || i == n - 1;
      if (first) ++seg;
      // (1) drain this CTA's partial Z of the tile
      if (!__all_sync(0xffffffffu, mbar_wait(&zacc_full[s], (i >> 1) & 1, a.status))) { ok = false; break; }
      fence_after();
      float z[16];
      tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + zacc_col(s), z);
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&zacc_empty[s]);
      if (nk == 0)
#pragma unroll
        for (int k = 0; k < 16; ++k) z[k] = 0.f;
      // (2) send the row to its owner once every owner has released zred
      if (i >= 1 && !__all_sync(0xffffffffu, mbar_wait(&rfull[(i - 1) & 1], ((i - 1) >> 1) & 1, a.status))) {
        ok = false;
        break;
      }
#pragma unroll
      for (int v = 0; v < 4; ++v)
        st_async_v4(zred_remote + v * 16, make_float4(z[4 * v], z[4 * v + 1], z[4 * v + 2], z[4 * v + 3]), zbar_remote);
      // (3) own rows: sum the 8 slices, softmax, R block to every CTA
      if (!__all_sync(0xffffffffu, mbar_wait_cluster(zred_full, i & 1, a.status))) { ok = false; break; }
      float2 zz = make_float2(0.f, 0.f);
#pragma unroll
      for (int src = 0; src < kCS; ++src) {
        const float2 v = *reinterpret_cast<const float2*>(zred + src * (16 * kNC) + j * kNC + 2 * cp);
        zz.x += v.x;
        zz.y += v.y;
      }
      named_sync(1, 128);                         // every reader is done with zred
      if (t == 0 && i + 1 < n) mbar_arrive_expect_tx(zred_full, kCS * kZPart);
      const int k0 = 2 * cp, k1 = 2 * cp + 1;
      const float za = k0 < a.K ? zz.x : -INFINITY, zb = k1 < a.K ? zz.y : -INFINITY;
      float m = fmaxf(za, zb);
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      const float ea = k0 < a.K ? expf(za - m) : 0.f, eb = k1 < a.K ? expf(zb - m) : 0.f;
      float sum = ea + eb;
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      const int tr = (int)rank * 16 + j;          // tile row
      const bool valid = tr < tl.y;
      const int lab = valid ? a.y[tl.x + tr] : -1;
      const float inv = 1.0f / sum;
      const float ra = valid && k0 < a.K ? ea * inv - (k0 == lab ? 1.f : 0.f) : 0.f;
      const float rb = valid && k1 < a.K ? eb * inv - (k1 == lab ? 1.f : 0.f) : 0.f;
      uint8_t* blk = rstage + 2 * s * kRBlock;
      uint8_t* blk_lo = blk + kRBlock;
      {
        const __nv_bfloat16 ha = __float2bfloat16_rn(ra), hb = __float2bfloat16_rn(rb);
        *reinterpret_cast<__nv_bfloat16*>(blk + r_offset(k0, j)) = ha;
        *reinterpret_cast<__nv_bfloat16*>(blk + r_offset(k1, j)) = hb;
        *reinterpret_cast<__nv_bfloat16*>(blk_lo + r_offset(k0, j)) = __float2bfloat16_rn(ra - __bfloat162float(ha));
        *reinterpret_cast<__nv_bfloat16*>(blk_lo + r_offset(k1, j)) = __float2bfloat16_rn(rb - __bfloat162float(hb));
      }
      fence_proxy_async_smem();
      named_sync(1, 128);
      if (t == 0) {
        const uint32_t dst_off = smem_u32(rbuf + s * kCS * kRBlock) + rank * kRBlock;
        const uint32_t dst_lo = smem_u32(rbuf_lo + s * kCS * kRBlock) + rank * kRBlock;
        for (uint32_t d = 0; d < (uint32_t)kCS; ++d) {
          bulk_s2cluster(mapa(dst_off, d), blk, kRBlock, mapa(smem_u32(&rfull[s]), d));
          bulk_s2cluster(mapa(dst_lo, d), blk_lo, kRBlock, mapa(smem_u32(&rfull[s]), d));
        }
      }
      // (4) end of this cluster's run in a partition: write the G^T slices
      if (last) {
        const int g = seg & 1;
        if (!__all_sync(0xffffffffu, mbar_wait(&gfull[g], (seg >> 1) & 1, a.status))) { ok = false; break; }
        fence_after();
        if (!waited) { grid_dep_wait(); waited = true; }   // partials of the previous step are consumed
        float* dst = a.partials + (int64_t)tl.z * a.P;
        for (int mt = 0; mt < nmt; ++mt) {
          float gv[16];
          tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + gacc_col(g) + mt * kNC, gv);
          const int f = (kb0 + 2 * mt) * 64 + q * 32 + lane;
          if (f < (kb0 + nk) * 64) {
#pragma unroll
            for (int k = 0; k < kNC; ++k)
              if (k < a.K) dst[(int64_t)k * a.ld + f] = gv[k];
          }
        }
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&gempty[g]);
      }
    }
    if (!ok) atomicExch(&cta_err, 1);
  }
  if (warp == 1 && lane == 0) {
    // every MMA issued by this CTA has completed before TMEM is released
    commit(mma_done);
    mbar_wait(mma_done, 0, a.status);
  }
  __syncthreads();
  fence_before();
  cl_sync();                          // no peer still sends into this CTA
  fence_after();
  if (warp == 1) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

int smallk_max_clusters(int nper) {
  const SkSmem L = sk_smem(nper);
  const size_t smem = 1024 + L.total;
  if (cudaFuncSetAttribute(softmax_smallk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCS);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int nc = 0;
  if (cudaOccupancyMaxActiveClusters(&nc, softmax_smallk_kernel, &cfg) != cudaSuccess) return 0;
  return nc;
}

bool smallk_fits(int64_t K, int64_t ld) {
  const int64_t nkb = ld / 64;
  const int64_t nper = (nkb + kCS - 1) / kCS;
  return K <= kNC && ld % 64 == 0 && nper >= 1 && sk_smem((int)nper).total + 1024 + 1024 <= 232448;
}

cudaError_t launch_softmax_smallk(const void* tmX, const void* tmW, const SmallKArgs& a, int nclusters,
                                  cudaStream_t st) {
  if (nclusters < 1) return cudaErrorInvalidValue;
  const SkSmem L = sk_smem(a.nper);
  const size_t smem = 1024 + L.total;
  cudaError_t e = cudaFuncSetAttribute(softmax_smallk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(kCS * nclusters));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.pdl ? 2 : 1;
  CUtensorMap x, w;
  std::memcpy(&x, tmX, sizeof(CUtensorMap));
  std::memcpy(&w, tmW, sizeof(CUtensorMap));
  return cudaLaunchKernelEx(&cfg, softmax_smallk_kernel, x, w, a);
}

}  // namespace pgc
