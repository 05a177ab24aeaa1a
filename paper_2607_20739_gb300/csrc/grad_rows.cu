// K1 — per-partition gradient of logistic and least-squares losses, one pass
// over the features (§III: g_k = (1/m_k) sum_{x in D_k} grad f; the 1/m_k is
// applied by the commit kernel).
//
// Each CTA streams one work item (a contiguous row range of one partition)
// from HBM into shared memory with 1-D bulk async copies (one producer
// thread, a ring of S stages, mbarrier full/empty handshakes).  Every row is
// read from HBM once: it is dotted with w, turned into the residual
// r = sigmoid(x.w) - y (logistic) or x.w - y (least squares), and
// accumulated as r * x, all while it sits in shared memory.
//
//   warp-row  (row <= 1024 fp32 / 2048 bf16 elements): one warp per row; each
//             lane holds NCH chunks of VEC elements of the row, of w and of
//             its gradient accumulator; the dot is a warp-shuffle sum.  The
//             8 warps' accumulators are summed in a fixed order at the end.
//   block-row (longer rows): all 256 consumer threads share each row; each
//             thread owns NCH chunks of columns; the dot is a shuffle sum
//             plus one shared-memory exchange per stage.
//
// Output: partial[item][0:ld] = sum over the item's rows of r * x (fp32).
#include "dev_common.cuh"
#include "pgc_internal.h"
#include "../../include/pgc.h"

namespace pgc {

constexpr int kNW = 8;                 // consumer warps per CTA
constexpr int kNT = kNW * 32;          // consumer threads
constexpr int kThreads = kNT + 32;     // + one producer warp
constexpr int kMaxItemRows = 8192;     // labels of one item staged in smem

struct StageCfg {
  int SR;            // rows per stage
  int S;             // stages
  uint32_t stage_bytes;
  size_t smem;       // dynamic shared memory
};

__device__ __forceinline__ float residual(int loss, float z, float y) {
  return loss == PGC_LOGISTIC ? 1.0f / (1.0f + expf(-z)) - y : z - y;
}

// Shared-memory map: [2S mbarriers | labels | (block-row: dot exchange) | stages]
struct SmemMap {
  uint64_t* full;
  uint64_t* empty;
  float* ylab;
  float* xdot;
  uint8_t* stages;
};

__device__ __forceinline__ SmemMap carve(uint8_t* smem, int S, int max_rows, int SR, bool block_row) {
  SmemMap m;
  m.full = reinterpret_cast<uint64_t*>(smem);
  m.empty = m.full + S;
  size_t off = 128;
  m.ylab = reinterpret_cast<float*>(smem + off);
  off += ((size_t)max_rows * 4 + 127) & ~size_t(127);
  m.xdot = reinterpret_cast<float*>(smem + off);
  if (block_row) off += ((size_t)2 * SR * kNW * 4 + 127) & ~size_t(127);
  m.stages = smem + off;
  return m;
}

// Producer: stream `nst` stages of the item's rows; afterwards wait until
// every issued copy has landed so no copy outlives the CTA.
__device__ __forceinline__ void produce(const SmemMap& sm, const uint8_t* src, int64_t rows, int64_t rb,
                                        int SR, int S, uint32_t stage_bytes, int* status) {
  const uint64_t pol = policy_evict_first();
  const int nst = (int)((rows + SR - 1) / SR);
  int issued = 0;
  for (int i = 0; i < nst; ++i) {
    const int s = i % S;
    if (i >= S && !mbar_wait(&sm.empty[s], ((i / S) - 1) & 1, status)) break;
    const int64_t r = rows - (int64_t)i * SR < SR ? rows - (int64_t)i * SR : SR;
    const uint32_t bytes = (uint32_t)(r * rb);
    mbar_arrive_expect_tx(&sm.full[s], bytes);
    bulk_g2s_stream(sm.stages + (size_t)s * stage_bytes, src + (size_t)i * SR * rb, bytes, &sm.full[s], pol);
    issued = i + 1;
  }
  for (int s = 0; s < S && s < issued; ++s) {
    const int last = ((issued - 1 - s) / S) * S + s;
    mbar_wait(&sm.full[s], (last / S) & 1, status);
  }
}

template <typename T, int VEC, int NCH>
__global__ void __launch_bounds__(kThreads, 1)
grad_rows_warp(GradRowsArgs a, int SR, int S, uint32_t stage_bytes, int max_rows) {
  extern __shared__ __align__(128) uint8_t smem[];
  using V = Vec<T, VEC>;
  constexpr int E = NCH * VEC;
  const SmemMap sm = carve(smem, S, max_rows, SR, false);
  const WorkItem it = a.items[blockIdx.x];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t rb = a.ld * (int64_t)sizeof(T);
  const int nst = (int)((it.rows + SR - 1) / SR);
  __shared__ int cta_err;

  if (threadIdx.x == 0) {
    cta_err = 0;
    for (int s = 0; s < S; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kNW);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kNW) {
    if (lane == 0)
      produce(sm, reinterpret_cast<const uint8_t*>(a.X) + it.row0 * rb, it.rows, rb, SR, S, stage_bytes,
              a.status);
  } else {
    // labels of the whole item, and this lane's slice of w
    for (int64_t r = threadIdx.x; r < it.rows; r += kNT) sm.ylab[r] = a.y[it.row0 + r];
    float wr[E], acc[E];
#pragma unroll
    for (int j = 0; j < NCH; ++j)
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        wr[j * VEC + v] = a.w[(j * 32 + lane) * VEC + v];
        acc[j * VEC + v] = 0.f;
      }
    named_bar_sync(1, kNT);
    bool ok = true;
    for (int i = 0; i < nst && ok; ++i) {
      const int s = i % S;
      const bool got = mbar_wait(&sm.full[s], (i / S) & 1, a.status);
      if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
      const int64_t rows_i = it.rows - (int64_t)i * SR < SR ? it.rows - (int64_t)i * SR : SR;
      const uint8_t* st = sm.stages + (size_t)s * stage_bytes;
      for (int rr = warp; rr < rows_i; rr += kNW) {
        const typename V::raw* row = reinterpret_cast<const typename V::raw*>(st + rr * rb);
        float x[E];
#pragma unroll
        for (int j = 0; j < NCH; ++j) V::widen(row[j * 32 + lane], &x[j * VEC]);
        float dot = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e) dot = fmaf(x[e], wr[e], dot);
        dot = warp_sum(dot);
        const float r = residual(a.loss, dot, sm.ylab[(int64_t)i * SR + rr]);
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] = fmaf(r, x[e], acc[e]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[s]);
    }
    if (!ok) atomicExch(&cta_err, 1);
    named_bar_sync(1, kNT);
    if (!cta_err) {
      // every stage was consumed, so no copy is in flight: reuse the stages
      float* red = reinterpret_cast<float*>(sm.stages);
#pragma unroll
      for (int j = 0; j < NCH; ++j)
#pragma unroll
        for (int v = 0; v < VEC; ++v) red[(size_t)warp * a.ld + (j * 32 + lane) * VEC + v] = acc[j * VEC + v];
      named_bar_sync(1, kNT);
      float* out = a.partials + (size_t)blockIdx.x * a.ld;
      for (int64_t col = threadIdx.x; col < a.ld; col += kNT) {
        float sum = 0.f;
#pragma unroll
        for (int w8 = 0; w8 < kNW; ++w8) sum += red[(size_t)w8 * a.ld + col];
        out[col] = sum;
      }
    }
  }
  __syncthreads();
}

template <typename T, int VEC, int NCH>
__global__ void __launch_bounds__(kThreads, 1)
grad_rows_block(GradRowsArgs a, int SR, int S, uint32_t stage_bytes, int max_rows) {
  extern __shared__ __align__(128) uint8_t smem[];
  using V = Vec<T, VEC>;
  constexpr int E = NCH * VEC;
  const SmemMap sm = carve(smem, S, max_rows, SR, true);
  const WorkItem it = a.items[blockIdx.x];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tid = threadIdx.x;
  const int64_t rb = a.ld * (int64_t)sizeof(T);
  const int nst = (int)((it.rows + SR - 1) / SR);
  __shared__ int cta_err;

  if (threadIdx.x == 0) {
    cta_err = 0;
    for (int s = 0; s < S; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kNW);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kNW) {
    if (lane == 0)
      produce(sm, reinterpret_cast<const uint8_t*>(a.X) + it.row0 * rb, it.rows, rb, SR, S, stage_bytes,
              a.status);
  } else {
    for (int64_t r = tid; r < it.rows; r += kNT) sm.ylab[r] = a.y[it.row0 + r];
    float wr[E], acc[E];
#pragma unroll
    for (int j = 0; j < NCH; ++j)
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        wr[j * VEC + v] = a.w[(j * kNT + tid) * VEC + v];
        acc[j * VEC + v] = 0.f;
      }
    named_bar_sync(1, kNT);
    bool ok = true;
    for (int i = 0; i < nst; ++i) {
      const int s = i % S;
      // Every consumer warp runs all nst iterations and reaches every named
      // barrier; once a wait has timed out the warp only skips its waits and
      // arithmetic, and the CTA's result is dropped at the end.
      if (ok && !__all_sync(0xffffffffu, mbar_wait(&sm.full[s], (i / S) & 1, a.status))) {
        ok = false;
        if (lane == 0) atomicExch(&cta_err, 1);
      }
      const int rows_i = (int)(it.rows - (int64_t)i * SR < SR ? it.rows - (int64_t)i * SR : SR);
      const uint8_t* st = sm.stages + (size_t)s * stage_bytes;
      float* xd = sm.xdot + (size_t)(i & 1) * SR * kNW;
      for (int rr = 0; rr < rows_i; ++rr) {
        float dot = 0.f;
        if (ok) {
          const typename V::raw* row = reinterpret_cast<const typename V::raw*>(st + rr * rb);
#pragma unroll
          for (int j = 0; j < NCH; ++j) {
            float x[VEC];
            V::widen(row[j * kNT + tid], x);
#pragma unroll
            for (int v = 0; v < VEC; ++v) dot = fmaf(x[v], wr[j * VEC + v], dot);
          }
        }
        dot = warp_sum(dot);
        if (lane == 0) xd[rr * kNW + warp] = dot;
      }
      named_bar_sync(1, kNT);
      if (ok) {
        for (int rr = 0; rr < rows_i; ++rr) {
          float dot = 0.f;
#pragma unroll
          for (int w8 = 0; w8 < kNW; ++w8) dot += xd[rr * kNW + w8];
          const float r = residual(a.loss, dot, sm.ylab[(int64_t)i * SR + rr]);
          const typename V::raw* row = reinterpret_cast<const typename V::raw*>(st + rr * rb);
#pragma unroll
          for (int j = 0; j < NCH; ++j) {
            float x[VEC];
            V::widen(row[j * kNT + tid], x);
#pragma unroll
            for (int v = 0; v < VEC; ++v) acc[j * VEC + v] = fmaf(r, x[v], acc[j * VEC + v]);
          }
        }
      }
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(&sm.empty[s]);
    }
    named_bar_sync(1, kNT);
    if (!cta_err) {
      float* out = a.partials + (size_t)blockIdx.x * a.ld;
#pragma unroll
      for (int j = 0; j < NCH; ++j)
#pragma unroll
        for (int v = 0; v < VEC; ++v) out[(j * kNT + tid) * VEC + v] = acc[j * VEC + v];
    }
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

static StageCfg stage_cfg(int variant, int64_t ld, int max_rows) {
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
  size_t fixed = 128 + (((size_t)max_rows * 4 + 127) & ~size_t(127));
  if (block) fixed += ((size_t)2 * c.SR * kNW * 4 + 127) & ~size_t(127);
  const size_t budget = 200 * 1024;
  int S = (int)((budget - fixed) / c.stage_bytes);
  c.S = S > 8 ? 8 : S;
  c.smem = fixed + (size_t)c.S * c.stage_bytes;
  // the warp-row epilogue reuses the stages for kNW * ld fp32 values
  return c;
}

int grad_rows_stage_rows(int variant, int64_t ld, int dtype) {
  (void)dtype;
  return stage_cfg(variant, ld, 1).SR;
}

template <typename K>
static cudaError_t launch_k(K kern, const GradRowsArgs& a, const StageCfg& c, int max_rows, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)c.smem);
  if (e != cudaSuccess) return e;
  kern<<<a.nitems, kThreads, c.smem, st>>>(a, c.SR, c.S, c.stage_bytes, max_rows);
  return cudaGetLastError();
}

#define PGC_WR(T, VEC, NCH) grad_rows_warp<T, VEC, NCH>
#define PGC_BR(T, VEC, NCH) grad_rows_block<T, VEC, NCH>

cudaError_t launch_grad_rows(const GradRowsArgs& a, int variant, cudaStream_t st) {
  if (a.nitems <= 0) return cudaSuccess;
  // the largest item decides the label buffer; the host caps items
  const int max_rows = a.max_item_rows;
  if (max_rows < 1 || max_rows > kMaxItemRows) return cudaErrorInvalidValue;
  const StageCfg c = stage_cfg(variant, a.ld, max_rows);
  if (c.S < 2) return cudaErrorInvalidValue;
  switch (variant) {
    // warp-row fp32: VEC 1,2,4 (NCH 1) and VEC 4 with NCH 2..8
    case 0 * 8 + 0: return launch_k(PGC_WR(float, 1, 1), a, c, max_rows, st);
    case 1 * 8 + 0: return launch_k(PGC_WR(float, 2, 1), a, c, max_rows, st);
    case 2 * 8 + 0: return launch_k(PGC_WR(float, 4, 1), a, c, max_rows, st);
    case 2 * 8 + 1: return launch_k(PGC_WR(float, 4, 2), a, c, max_rows, st);
    case 2 * 8 + 2: return launch_k(PGC_WR(float, 4, 4), a, c, max_rows, st);
    case 2 * 8 + 3: return launch_k(PGC_WR(float, 4, 8), a, c, max_rows, st);
    // warp-row bf16: VEC 2,4,8 (NCH 1) and VEC 8 with NCH 2..8
    case 32 + 1 * 8 + 0: return launch_k(PGC_WR(uint16_t, 2, 1), a, c, max_rows, st);
    case 32 + 2 * 8 + 0: return launch_k(PGC_WR(uint16_t, 4, 1), a, c, max_rows, st);
    case 32 + 3 * 8 + 0: return launch_k(PGC_WR(uint16_t, 8, 1), a, c, max_rows, st);
    case 32 + 3 * 8 + 1: return launch_k(PGC_WR(uint16_t, 8, 2), a, c, max_rows, st);
    case 32 + 3 * 8 + 2: return launch_k(PGC_WR(uint16_t, 8, 4), a, c, max_rows, st);
    case 32 + 3 * 8 + 3: return launch_k(PGC_WR(uint16_t, 8, 8), a, c, max_rows, st);
    // block-row fp32 (VEC 4) and bf16 (VEC 8), NCH 1..16
    case 64 + 2 * 8 + 0: return launch_k(PGC_BR(float, 4, 1), a, c, max_rows, st);
    case 64 + 2 * 8 + 1: return launch_k(PGC_BR(float, 4, 2), a, c, max_rows, st);
    case 64 + 2 * 8 + 2: return launch_k(PGC_BR(float, 4, 4), a, c, max_rows, st);
    case 64 + 2 * 8 + 3: return launch_k(PGC_BR(float, 4, 8), a, c, max_rows, st);
    case 64 + 2 * 8 + 4: return launch_k(PGC_BR(float, 4, 16), a, c, max_rows, st);
    case 64 + 32 + 3 * 8 + 0: return launch_k(PGC_BR(uint16_t, 8, 1), a, c, max_rows, st);
    case 64 + 32 + 3 * 8 + 1: return launch_k(PGC_BR(uint16_t, 8, 2), a, c, max_rows, st);
    case 64 + 32 + 3 * 8 + 2: return launch_k(PGC_BR(uint16_t, 8, 4), a, c, max_rows, st);
    case 64 + 32 + 3 * 8 + 3: return launch_k(PGC_BR(uint16_t, 8, 8), a, c, max_rows, st);
    case 64 + 32 + 3 * 8 + 4: return launch_k(PGC_BR(uint16_t, 8, 16), a, c, max_rows, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace pgc
