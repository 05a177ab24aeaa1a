// K1 — per-partition gradient of logistic and least-squares losses, one pass
// over the features (§III: g_k = (1/m_k) sum_{x in D_k} grad f; the 1/m_k is
// applied when the partition is committed).
//
// Work: the evaluated partitions' rows are cut into work items (contiguous
// row ranges of one partition).  A persistent grid (at most one CTA per SM)
// takes items dynamically: item blockIdx.x first, then the next free index
// from a device counter, so SMs that stream faster take more items.  Each
// item's sum over its rows of r(x) * x goes to its own partial slot, so the
// result does not depend on which CTA took which item.
//
// Per CTA: one producer thread streams each item's rows from HBM into a ring
// of S shared-memory stages with 1-D bulk async copies (rows and their labels,
// completion counted on the stage's mbarrier); 8 consumer warps dot each row
// with w, form the residual r = sigmoid(x.w) - y (logistic) or x.w - y (least
// squares) and accumulate r * x while the row sits in shared memory, so every
// feature byte is read from HBM once.
//   warp-row  (row <= 1024 fp32 / 2048 bf16 elements): one warp per row; each
//             lane holds NCH chunks of VEC elements of the row, of w and of
//             its accumulator; the dot is a warp-shuffle sum; at the end of an
//             item the 8 warps' accumulators are summed in a fixed order.
//   block-row (longer rows): the 256 consumer threads share each row; each
//             owns NCH chunks of columns; the dots of a stage are exchanged
//             once through shared memory.
//
// Item ends: consumers hand their accumulators to a tail warp (through a
// shared buffer and two mbarriers) and keep streaming.  The tail warp sums the
// 8 warps' accumulators in a fixed order into the item's partial slot and,
// with tail >= 1, counts the item for its partition.  When that count
// completes a partition, the consumers commit it at their next item end (or
// after their last item): ordered sum of the partition's partials, scaled by
// 1/m, into its destination stores.  With tail == 2 the CTA that commits the
// last partition also derives the decode coefficients from the mask, decodes
// and applies the SGD update.
//
// Programmatic dependent launch: the producer streams its first item before
// waiting for the previous step's kernel; consumers wait before reading w.
//
// Every wait is bounded (mbarrier try_wait with an iteration and time limit).
// Consumer warps synchronise through mbarriers, never named barriers, so a
// wait that gives up cannot leave another warp blocked: the CTA then skips
// its remaining work, flags the status word and exits.
#include "tail.cuh"

namespace pgc {

constexpr int kNW = 8;                 // consumer warps per CTA
constexpr int kNT = kNW * 32;          // consumer threads
constexpr int kThreads = kNT + 64;     // + a producer warp + a tail warp
constexpr int kProducer = kNT;        // producer thread
constexpr int kTailWarp = kNW + 1;     // warp index of the tail warp
constexpr int64_t kPrefetchChunkRows = 16;

struct StageHdr {
  int item;      // work item, or -1: no more work
  int e;         // evaluated-partition position of the item
  int rows;      // rows in this stage
  int lab_off;   // index of the stage's first label in its label slot
  int last;      // last stage of the item
  int pad[3];
};

struct StageCfg {
  int SR;              // rows per stage
  int S;               // stages
  uint32_t stage_bytes;
  int LS;              // floats per label slot
  size_t red_bytes;    // item-end reduction buffer
  size_t plan_bytes;   // decode plan (fused decode only)
  size_t smem;         // dynamic shared memory
};

__device__ __forceinline__ float residual(int loss, float z, float y) {
  return loss == PGC_LOGISTIC ? 1.0f / (1.0f + expf(-z)) - y : z - y;
}

// Item handoff between the consumers and the tail warp.
struct Handoff {
  int item;            // item whose accumulators are in red, or -1: no more items
  int e;
  int commit;          // set by the tail warp: partition to commit, or -1
  int decode;          // set by the consumers: this CTA decodes
  unsigned sync_count; // arrivals at the consumer barrier (ConsumerSync)
};

// Shared memory: [full S | empty S | sync, red_full, red_free, tail_done]
//                [handoff] [S headers] [S label slots] [red / decode scratch]
//                [dot exchange] [S stages]
struct Smem {
  uint64_t* full;
  uint64_t* empty;
  uint64_t* sync;       // consumer barrier (count kNW)
  uint64_t* red_full;   // consumers -> tail warp (count kNW)
  uint64_t* red_free;   // tail warp -> consumers (count 1)
  uint64_t* stage_sync; // CTA-per-row dot exchange (count kNW)
  Handoff* ho;
  DecodePlan* plan;     // decode coefficients (tail == 2), derived at kernel start
  StageHdr* hdr;
  float* lab;
  uint8_t* red;
  float* xdot;
  uint8_t* stages;
};

__host__ __device__ inline size_t a128(size_t v) { return (v + 127) & ~size_t(127); }

__host__ __device__ inline size_t fixed_bytes(int S, int LS, size_t red, int SR, bool block_row, size_t plan) {
  return a128(sizeof(uint64_t) * (2 * S + 4)) + a128(sizeof(Handoff)) + a128(plan) + a128(sizeof(StageHdr) * S) +
         a128(sizeof(float) * LS * S) + a128(red) + (block_row ? a128(sizeof(float) * 2 * SR * kNW) : 0);
}

__device__ __forceinline__ Smem carve(uint8_t* base, const StageCfg& c, bool block_row) {
  Smem m;
  size_t off = 0;
  m.full = reinterpret_cast<uint64_t*>(base);
  m.empty = m.full + c.S;
  m.sync = m.empty + c.S;
  m.red_full = m.sync + 1;
  m.red_free = m.sync + 2;
  m.stage_sync = m.sync + 3;
  off = a128(sizeof(uint64_t) * (2 * c.S + 4));
  m.ho = reinterpret_cast<Handoff*>(base + off);
  off = a128(off + sizeof(Handoff));
  m.plan = reinterpret_cast<DecodePlan*>(base + off);
  off = a128(off + c.plan_bytes);
  m.hdr = reinterpret_cast<StageHdr*>(base + off);
  off = a128(off + sizeof(StageHdr) * c.S);
  m.lab = reinterpret_cast<float*>(base + off);
  off = a128(off + sizeof(float) * c.LS * c.S);
  m.red = base + off;
  off = a128(off + c.red_bytes);
  m.xdot = reinterpret_cast<float*>(base + off);
  if (block_row) off = a128(off + sizeof(float) * 2 * c.SR * kNW);
  m.stages = base + off;
  return m;
}

// A barrier of the 8 consumer warps on an mbarrier (count kNW), bounded.
// Each warp also counts its arrival on a shared counter; the warp whose
// arrival is the kNW-th knows every other warp is already through its
// pre-barrier work and does not wait (waiting on a phase it completed itself
// was measured to cost microseconds).
struct ConsumerSync {
  uint64_t* bar;
  unsigned* count;
  uint32_t phase;
  int* status;
  __device__ __forceinline__ bool operator()() {
    __syncwarp();
    int last = 0;
    if ((threadIdx.x & 31) == 0) {
      last = (atomic_add_cta_acq_rel(count, 1u) + 1u) % (unsigned)kNW == 0u;
      mbar_arrive(bar);
    }
    last = __shfl_sync(0xffffffffu, last, 0);
    __syncwarp();                        // lane 0's acquire covers the whole warp
    bool ok = true;
    if (!last) ok = mbar_wait(bar, phase, status);
    phase ^= 1u;
    return __all_sync(0xffffffffu, ok);
  }
};

// A plain barrier of the 8 consumer warps on its own mbarrier (count kNW),
// bounded: used once per stage by the CTA-per-row consumers, where every
// warp arrives at about the same time.
struct StageSync {
  uint64_t* bar;
  uint32_t phase;
  int* status;
  __device__ __forceinline__ bool operator()() {
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
    const bool ok = mbar_wait(bar, phase, status);
    phase ^= 1u;
    return __all_sync(0xffffffffu, ok);
  }
};

// ---------------------------------------------------------------------------
// producer
// ---------------------------------------------------------------------------
__device__ void produce(const GradRowsArgs& a, const Smem& sm, const StageCfg& c, int64_t rb) {
  const uint64_t pol = policy_evict_first();
  const uint8_t* X = static_cast<const uint8_t*>(a.X);
  const uint8_t* Y = reinterpret_cast<const uint8_t*>(a.y);
  int i = 0;                     // stages issued
  bool ok = true, waited = false;
  int item = blockIdx.x;
  if (item < a.nitems) {
    // Beyond the S stages it can hold, optionally warm L2 with the next rows
    // of the first item while the previous step finishes (a.prefetch_bytes;
    // on the streaming workloads this traffic slowed the previous step's
    // serial tail more than it saved, so the library passes 0).
    const WorkItem it = a.items[item];
    const int64_t r0 = it.row0 + (int64_t)c.S * c.SR;
    int64_t rows = it.rows - (int64_t)c.S * c.SR;
    const int64_t cap = a.prefetch_bytes / rb;
    rows = rows < cap ? rows : cap;
    for (int64_t r = 0; r < rows; r += kPrefetchChunkRows) {
      const int64_t n = rows - r < kPrefetchChunkRows ? rows - r : kPrefetchChunkRows;
      prefetch_l2(X + (r0 + r) * rb, (uint32_t)(n * rb));
    }
  }
  while (ok && item < a.nitems) {
    const WorkItem it = a.items[item];
    const int nst = (int)((it.rows + c.SR - 1) / c.SR);
    for (int j = 0; j < nst; ++j) {
      const int s = i % c.S;
      if (i >= c.S && !mbar_wait(&sm.empty[s], ((i / c.S) - 1) & 1, a.status)) { ok = false; break; }
      const int64_t r0 = it.row0 + (int64_t)j * c.SR;
      const int rows = (int)(it.rows - (int64_t)j * c.SR < c.SR ? it.rows - (int64_t)j * c.SR : c.SR);
      const int64_t la = r0 & ~int64_t(3);                      // 16-byte aligned label start
      const uint32_t lbytes = (uint32_t)(((r0 + rows - la) * 4 + 15) & ~int64_t(15));
      StageHdr h;
      h.item = item; h.e = it.e; h.rows = rows; h.lab_off = (int)(r0 - la); h.last = j == nst - 1;
      sm.hdr[s] = h;
      const uint32_t xbytes = (uint32_t)(rows * rb);
      mbar_arrive_expect_tx(&sm.full[s], xbytes + lbytes);
      bulk_g2s_stream(sm.stages + (size_t)s * c.stage_bytes, X + r0 * rb, xbytes, &sm.full[s], pol);
      bulk_g2s(sm.lab + (size_t)s * c.LS, Y + la * 4, lbytes, &sm.full[s]);
      ++i;
    }
    if (!ok || !a.work_ctr) break;
    if (a.pdl && !waited) { grid_dep_wait(); waited = true; }   // counters belong to the previous step until now
    item = (int)gridDim.x + atomicAdd(a.work_ctr, 1);
  }
  if (ok) {   // end marker: a stage without data
    const int s = i % c.S;
    if (i < c.S || mbar_wait(&sm.empty[s], ((i / c.S) - 1) & 1, a.status)) {
      sm.hdr[s].item = -1;
      mbar_arrive(&sm.full[s]);
      ++i;
    }
  }
  if (a.work_ctr) {
    if (a.pdl && !waited) grid_dep_wait();
    // the last producer to finish resets the item counter for the next step
    if (atomicAdd(a.prod_done, 1) == (int)gridDim.x - 1) {
      *a.work_ctr = 0;
      *a.prod_done = 0;
    }
  }
  // no copy may outlive the CTA: wait for the last use of every stage
  for (int s = 0; s < c.S && s < i; ++s) {
    const int last = ((i - 1 - s) / c.S) * c.S + s;
    mbar_wait(&sm.full[s], (last / c.S) & 1, a.status);
  }
}

// ---------------------------------------------------------------------------
// tail warp: per-item reduction and partition counting
// ---------------------------------------------------------------------------
__device__ void tail_warp(const GradRowsArgs& a, const Smem& sm, bool warp_row) {
  const int lane = threadIdx.x & 31;
  if (a.tail == 2) derive_plan_warp(a.dec, *sm.plan, lane);   // depends only on the mask
  if (a.pdl) grid_dep_wait();          // partials and counters belong to the previous step until now
  const float* red = reinterpret_cast<const float*>(sm.red);
  for (uint32_t j = 0;; ++j) {
    if (!__all_sync(0xffffffffu, mbar_wait(sm.red_full, j & 1u, a.status))) break;
    const int item = sm.ho->item, e = sm.ho->e;
    if (item < 0) break;
    if (warp_row) {
      // fixed-order sum of the 8 warps' accumulators into the item's partial
      float4* out = reinterpret_cast<float4*>(a.partials + (size_t)item * a.ld);
      const float4* r4 = reinterpret_cast<const float4*>(red);
      const int64_t L4 = a.ld / 4;
      for (int64_t q = lane; q < L4; q += 32) {
        float4 acc = r4[q];
#pragma unroll
        for (int w8 = 1; w8 < kNW; ++w8) acc = f4add(acc, r4[(size_t)w8 * L4 + q]);
        out[q] = acc;
      }
    }
    int commit = -1;
    if (a.tail) {
      __syncwarp();
      if (lane == 0) {
        // release this item's partial (written by this warp, or by the
        // consumers before red_full) and acquire the other items' partials
        const int prev = atomic_add_acq_rel(&a.cnt_e[e], 1);
        if (prev == a.e_item0[e + 1] - a.e_item0[e] - 1) {
          a.cnt_e[e] = 0;              // every item of e has arrived: reset for the next step
          commit = e;
        }
      }
      commit = __shfl_sync(0xffffffffu, commit, 0);
    }
    if (lane == 0) {
      sm.ho->commit = commit;
      mbar_arrive(sm.red_free);
    }
    __syncwarp();
  }
}

// Consumers: commit partition e (all 256 consumer threads), then count it;
// the CTA completing the last partition decodes when tail == 2.
__device__ void consumer_commit(const GradRowsArgs& a, const Smem& sm, int e, int tid, ConsumerSync& bar, bool& ok) {
  // the tail warp acquired the other CTAs' partials (atomic + fence) before
  // handing e over through red_free
  commit_block(a.partials, a.ld, a.e_item0[e], a.e_item0[e + 1], a.e_scale[e], a.e_dest + (int64_t)e * a.ndest,
               a.ndest, a.store, tid, kNT);
  if (!bar()) { ok = false; return; }
  if (tid == 0) {
    // release the stores written by the whole CTA (ordered before this by the
    // barrier) and acquire the other committers' stores
    const bool all = atomic_add_acq_rel(a.cnt_all, 1) == a.nE - 1;
    if (all) *a.cnt_all = 0;
    if (all && a.tail == 2) sm.ho->decode = 1;
  }
}

__device__ void consumer_decode(const GradRowsArgs& a, const Smem& sm, int tid) {
  if (tid < 32) write_coeffs_warp(a.dec, tid);
  decode_columns(a.dec, *sm.plan, 0, a.dec.P / 4, tid, kNT);
}

// Item end, consumer side, called by all 8 warps at the same stage.
// handover_begin: wait until the tail warp has taken the previous item (so
// red and the handoff slot are free) and run the commit it asked for.
__device__ __forceinline__ bool handover_begin(const GradRowsArgs& a, const Smem& sm, uint32_t ends, ConsumerSync& bar,
                                               bool& ok) {
  if (ends == 0) return true;
  if (!__all_sync(0xffffffffu, mbar_wait(sm.red_free, (ends - 1) & 1u, a.status))) { ok = false; return false; }
  const int ce = sm.ho->commit;          // written by the tail warp before red_free: same for every warp
  if (ce >= 0) {
    consumer_commit(a, sm, ce, (int)threadIdx.x, bar, ok);
    if (!ok) return false;
  }
  return true;
}

// handover_end: publish the item (or -1: no more) to the tail warp.
__device__ __forceinline__ void handover_end(const Smem& sm, int item, int e, uint32_t& ends) {
  if (threadIdx.x == 0) { sm.ho->item = item; sm.ho->e = e; }
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(sm.red_full);
  ++ends;
}

// After the last item: final handoff, pending commit, decode if this CTA
// committed the last partition.
__device__ __forceinline__ void consumers_finish(const GradRowsArgs& a, const Smem& sm, uint32_t& ends,
                                                 ConsumerSync& bar, bool& ok) {
  if (ok && handover_begin(a, sm, ends, bar, ok)) {
    handover_end(sm, -1, -1, ends);
    if (!bar()) ok = false;              // the decode flag is written before this barrier
    if (ok && sm.ho->decode) consumer_decode(a, sm, (int)threadIdx.x);
  } else if (threadIdx.x < kNT) {
    // release the tail warp even on failure: it stops at item -1 or at its own bound
    handover_end(sm, -1, -1, ends);
  }
}

// ---------------------------------------------------------------------------
// consumers
// ---------------------------------------------------------------------------
template <typename T, int VEC, int NCH>
__device__ void consume_warp_row(const GradRowsArgs& a, const Smem& sm, const StageCfg& c, int64_t rb) {
  using V = Vec<T, VEC>;
  constexpr int E = NCH * VEC;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  ConsumerSync bar{sm.sync, &sm.ho->sync_count, 0u, a.status};
  if (a.pdl) grid_dep_wait();                       // w is the previous step's output
  float wr[E], acc[E];
#pragma unroll
  for (int j = 0; j < NCH; ++j)
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      wr[j * VEC + v] = a.w[(j * 32 + lane) * VEC + v];
      acc[j * VEC + v] = 0.f;
    }
  float* red = reinterpret_cast<float*>(sm.red);
  uint32_t ends = 0;
  bool ok = true;
  for (int i = 0; ok; ++i) {
    const int s = i % c.S;
    if (!__all_sync(0xffffffffu, mbar_wait(&sm.full[s], (i / c.S) & 1, a.status))) { ok = false; break; }
    const StageHdr h = sm.hdr[s];
    if (h.item < 0) break;
    const uint8_t* st = sm.stages + (size_t)s * c.stage_bytes;
    const float* lab = sm.lab + (size_t)s * c.LS + h.lab_off;
    for (int rr = warp; rr < h.rows; rr += kNW) {
      const typename V::raw* row = reinterpret_cast<const typename V::raw*>(st + rr * rb);
      float x[E];
#pragma unroll
      for (int j = 0; j < NCH; ++j) V::widen(row[j * 32 + lane], &x[j * VEC]);
      float dot = 0.f;
#pragma unroll
      for (int k = 0; k < E; ++k) dot = fmaf(x[k], wr[k], dot);
      dot = warp_sum(dot);
      const float r = residual(a.loss, dot, lab[rr]);
#pragma unroll
      for (int k = 0; k < E; ++k) acc[k] = fmaf(r, x[k], acc[k]);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.empty[s]);
    if (h.last) {
      if (!handover_begin(a, sm, ends, bar, ok)) break;
#pragma unroll
      for (int j = 0; j < NCH; ++j)
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          red[(size_t)warp * a.ld + (j * 32 + lane) * VEC + v] = acc[j * VEC + v];
          acc[j * VEC + v] = 0.f;
        }
      handover_end(sm, h.item, h.e, ends);
    }
  }
  consumers_finish(a, sm, ends, bar, ok);
  if (!ok) atomicOr(a.status, kErrWaitTimeout);
}

template <typename T, int VEC, int NCH>
__device__ void consume_block_row(const GradRowsArgs& a, const Smem& sm, const StageCfg& c, int64_t rb) {
  using V = Vec<T, VEC>;
  constexpr int E = NCH * VEC;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  ConsumerSync bar{sm.sync, &sm.ho->sync_count, 0u, a.status};
  StageSync xbar{sm.stage_sync, 0u, a.status};
  if (a.pdl) grid_dep_wait();
  float wr[E], acc[E];
#pragma unroll
  for (int j = 0; j < NCH; ++j)
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      wr[j * VEC + v] = a.w[(j * kNT + tid) * VEC + v];
      acc[j * VEC + v] = 0.f;
    }
  uint32_t ends = 0;
  bool ok = true;
  for (int i = 0; ok; ++i) {
    const int s = i % c.S;
    if (!__all_sync(0xffffffffu, mbar_wait(&sm.full[s], (i / c.S) & 1, a.status))) { ok = false; break; }
    const StageHdr h = sm.hdr[s];
    if (h.item < 0) break;
    const uint8_t* st = sm.stages + (size_t)s * c.stage_bytes;
    const float* lab = sm.lab + (size_t)s * c.LS + h.lab_off;
    float* xd = sm.xdot + (size_t)(i & 1) * c.SR * kNW;
    for (int rr = 0; rr < h.rows; ++rr) {
      const typename V::raw* row = reinterpret_cast<const typename V::raw*>(st + rr * rb);
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < NCH; ++j) {
        float x[VEC];
        V::widen(row[j * kNT + tid], x);
#pragma unroll
        for (int v = 0; v < VEC; ++v) dot = fmaf(x[v], wr[j * VEC + v], dot);
      }
      dot = warp_sum(dot);
      if (lane == 0) xd[rr * kNW + warp] = dot;
    }
    // the exchange buffer alternates by stage parity; the barrier of stage
    // i + 1 separates this stage's reads from stage i + 2's writes
    if (!xbar()) { ok = false; break; }
    for (int rr = 0; rr < h.rows; ++rr) {
      float dot = 0.f;
#pragma unroll
      for (int w8 = 0; w8 < kNW; ++w8) dot += xd[rr * kNW + w8];
      const float r = residual(a.loss, dot, lab[rr]);
      const typename V::raw* row = reinterpret_cast<const typename V::raw*>(st + rr * rb);
#pragma unroll
      for (int j = 0; j < NCH; ++j) {
        float x[VEC];
        V::widen(row[j * kNT + tid], x);
#pragma unroll
        for (int v = 0; v < VEC; ++v) acc[j * VEC + v] = fmaf(r, x[v], acc[j * VEC + v]);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.empty[s]);
    if (h.last) {
      if (!handover_begin(a, sm, ends, bar, ok)) break;
      // each thread owns its columns: write them straight to the item's partial
      float* out = a.partials + (size_t)h.item * a.ld;
#pragma unroll
      for (int j = 0; j < NCH; ++j)
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          out[(j * kNT + tid) * VEC + v] = acc[j * VEC + v];
          acc[j * VEC + v] = 0.f;
        }
      handover_end(sm, h.item, h.e, ends);
    }
  }
  consumers_finish(a, sm, ends, bar, ok);
  if (!ok) atomicOr(a.status, kErrWaitTimeout);
}

template <typename T, int VEC, int NCH, bool BLOCK>
__global__ void __launch_bounds__(kThreads, 1) grad_rows_kernel(GradRowsArgs a, StageCfg c) {
  extern __shared__ __align__(128) uint8_t smem[];
  const Smem sm = carve(smem, c, BLOCK);
  const int64_t rb = a.ld * (int64_t)sizeof(T);
  if (threadIdx.x == 0) {
    for (int s = 0; s < c.S; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kNW);
    }
    mbar_init(sm.sync, kNW);
    mbar_init(sm.red_full, kNW);
    mbar_init(sm.red_free, 1);
    mbar_init(sm.stage_sync, kNW);
    sm.ho->item = -1;
    sm.ho->e = -1;
    sm.ho->commit = -1;
    sm.ho->decode = 0;
    sm.ho->sync_count = 0;
    fence_mbar_init();
    grid_dep_launch();
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5;
  if (warp == kTailWarp) {
    tail_warp(a, sm, !BLOCK);
  } else if (threadIdx.x >= kNT) {
    if (threadIdx.x == kProducer) produce(a, sm, c, rb);
  } else if (BLOCK) {
    consume_block_row<T, VEC, NCH>(a, sm, c, rb);
  } else {
    consume_warp_row<T, VEC, NCH>(a, sm, c, rb);
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Variant table.  id = kind * 64 + dtype * 32 + log2(VEC) * 8 + log2(NCH)
// ---------------------------------------------------------------------------
namespace {
int ilog2(int v) { int l = 0; while ((1 << l) < v) ++l; return l; }
}

int grad_rows_variant(int dtype, int64_t d, int64_t* ld_out) {
  const int esz = dtype == PGC_BF16 ? 2 : 4;
  const int maxvec = 16 / esz;
  // warp-row: ld = 32 * VEC * NCH, VEC up to one 16-byte chunk, NCH up to 8
  for (int nch = 1; nch <= 8; nch *= 2) {
    for (int vec = 1; vec <= maxvec; vec *= 2) {
      if (dtype == PGC_BF16 && vec < 2) continue;
      if (nch > 1 && vec < maxvec) continue;
      const int64_t ld = 32LL * vec * nch;
      if (ld >= d) {
        *ld_out = ld;
        return 0 * 64 + (dtype == PGC_BF16) * 32 + ilog2(vec) * 8 + ilog2(nch);
      }
    }
  }
  // block-row: ld = 256 * VEC * NCH with full 16-byte chunks, NCH up to 16
  for (int nch = 1; nch <= 16; nch *= 2) {
    const int64_t ld = (int64_t)kNT * maxvec * nch;
    if (ld >= d) {
      *ld_out = ld;
      return 1 * 64 + (dtype == PGC_BF16) * 32 + ilog2(maxvec) * 8 + ilog2(nch);
    }
  }
  return -1;
}

static StageCfg stage_cfg(int variant, int64_t ld, int tail) {
  const bool block = variant >= 64;
  const int esz = (variant & 32) ? 2 : 4;
  const int64_t rb = ld * esz;
  StageCfg c;
  if (!block) {
    int rpw = (int)(32768 / (kNW * rb));
    rpw = rpw < 1 ? 1 : (rpw > 16 ? 16 : rpw);
    c.SR = kNW * rpw;
  } else {
    int sr = (int)(32768 / rb);
    c.SR = sr < 1 ? 1 : (sr > 8 ? 8 : sr);
  }
  c.stage_bytes = (uint32_t)(c.SR * rb);
  c.LS = ((c.SR + 3 + 3) / 4) * 4;   // labels of SR rows read from a 4-row-aligned start
  const size_t red = block ? 0 : (size_t)kNW * ld * sizeof(float);
  c.red_bytes = red;
  c.plan_bytes = tail == 2 ? sizeof(DecodePlan) : 0;
  const size_t budget = 220 * 1024;
  int S = 8;
  while (S > 2 && fixed_bytes(S, c.LS, red, c.SR, block, c.plan_bytes) + (size_t)S * c.stage_bytes > budget) --S;
  c.S = S;
  c.smem = fixed_bytes(S, c.LS, red, c.SR, block, c.plan_bytes) + (size_t)S * c.stage_bytes;
  return c;
}

int grad_rows_stage_rows(int variant, int64_t ld, int dtype) {
  (void)dtype;
  return stage_cfg(variant, ld, 0).SR;
}

template <typename K>
static cudaError_t launch_k(K kern, const GradRowsArgs& a, const StageCfg& c, int grid, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)c.smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = c.smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, a, c);
}

#define PGC_WR(T, VEC, NCH) grad_rows_kernel<T, VEC, NCH, false>
#define PGC_BR(T, VEC, NCH) grad_rows_kernel<T, VEC, NCH, true>

cudaError_t launch_grad_rows(const GradRowsArgs& a, int variant, cudaStream_t st) {
  if (a.nitems <= 0) return cudaSuccess;
  const StageCfg c = stage_cfg(variant, a.ld, a.tail);
  if (c.smem > 227 * 1024) return cudaErrorInvalidValue;
  // persistent grid when items are taken dynamically, else one CTA per item
  const int grid = a.work_ctr ? (a.grid < a.nitems ? a.grid : a.nitems) : a.nitems;
  if (grid < 1) return cudaErrorInvalidValue;
  switch (variant) {
    // warp-row fp32: VEC 1,2,4 (NCH 1) and VEC 4 with NCH 2..8
    case 0 * 8 + 0: return launch_k(PGC_WR(float, 1, 1), a, c, grid, st);
    case 1 * 8 + 0: return launch_k(PGC_WR(float, 2, 1), a, c, grid, st);
    case 2 * 8 + 0: return launch_k(PGC_WR(float, 4, 1), a, c, grid, st);
    case 2 * 8 + 1: return launch_k(PGC_WR(float, 4, 2), a, c, grid, st);
    case 2 * 8 + 2: return launch_k(PGC_WR(float, 4, 4), a, c, grid, st);
    case 2 * 8 + 3: return launch_k(PGC_WR(float, 4, 8), a, c, grid, st);
    // warp-row bf16: VEC 2,4,8 (NCH 1) and VEC 8 with NCH 2..8
    case 32 + 1 * 8 + 0: return launch_k(PGC_WR(uint16_t, 2, 1), a, c, grid, st);
    case 32 + 2 * 8 + 0: return launch_k(PGC_WR(uint16_t, 4, 1), a, c, grid, st);
    case 32 + 3 * 8 + 0: return launch_k(PGC_WR(uint16_t, 8, 1), a, c, grid, st);
    case 32 + 3 * 8 + 1: return launch_k(PGC_WR(uint16_t, 8, 2), a, c, grid, st);
    case 32 + 3 * 8 + 2: return launch_k(PGC_WR(uint16_t, 8, 4), a, c, grid, st);
    case 32 + 3 * 8 + 3: return launch_k(PGC_WR(uint16_t, 8, 8), a, c, grid, st);
    // block-row fp32 (VEC 4) and bf16 (VEC 8), NCH 1..16
    case 64 + 2 * 8 + 0: return launch_k(PGC_BR(float, 4, 1), a, c, grid, st);
    case 64 + 2 * 8 + 1: return launch_k(PGC_BR(float, 4, 2), a, c, grid, st);
    case 64 + 2 * 8 + 2: return launch_k(PGC_BR(float, 4, 4), a, c, grid, st);
    case 64 + 2 * 8 + 3: return launch_k(PGC_BR(float, 4, 8), a, c, grid, st);
    case 64 + 2 * 8 + 4: return launch_k(PGC_BR(float, 4, 16), a, c, grid, st);
    case 64 + 32 + 3 * 8 + 0: return launch_k(PGC_BR(uint16_t, 8, 1), a, c, grid, st);
    case 64 + 32 + 3 * 8 + 1: return launch_k(PGC_BR(uint16_t, 8, 2), a, c, grid, st);
    case 64 + 32 + 3 * 8 + 2: return launch_k(PGC_BR(uint16_t, 8, 4), a, c, grid, st);
    case 64 + 32 + 3 * 8 + 3: return launch_k(PGC_BR(uint16_t, 8, 8), a, c, grid, st);
    case 64 + 32 + 3 * 8 + 4: return launch_k(PGC_BR(uint16_t, 8, 16), a, c, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace pgc
