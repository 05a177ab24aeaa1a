// Host side of libpgc: argument checks, device state, the step schedule
// (§IV-A, §V-B), per-phase launch tables and the C ABI of include/pgc.h.
//
// Device state of a run (all owned by the context):
//   X      packed features [sum_k m_k][ld] (rows padded with zeros to ld)
//   y      packed labels [sum_k m_k] (float32, or int32 classes)
//   w      beta [K][ld] fp32 (+ a bf16 copy wb for bf16 features)
//   store  gradient stores [owners][c][K*ld] fp32: owners = n (CR) or n/c
//          (FR: the c members of a group keep identical stores, §IV-A)
//   U      slot totals [c][K*ld]: U[o] = sum over owners of store[.][o]
//   gout   decoded gradient of the last step [K*ld]
//
// Phases: phase 0 is the warm-up step t = 0 (every partition evaluated and
// written to all its holders); phase 1 + o is a steady step with
// o_t = (t - 1) mod c = o.  Each phase has a fixed list of evaluated
// partitions, the work items that split their rows across CTAs, and the
// destination stores of each new gradient.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "pgc.h"
#include "pgc_internal.h"

using namespace pgc;

namespace {

struct Phase {
  int slot = -1;                        // o, or -1 for the warm-up
  std::vector<int32_t> parts;           // evaluated partitions (e -> k)
  std::vector<WorkItem> items;          // row-kernel work items
  std::vector<int32_t> e_item0;         // CSR of items (or one per e)
  std::vector<float> e_scale;           // 1 / m_e
  std::vector<int32_t> e_dest;          // [nE * ndest] store index owner*c+slot
  int ndest = 1;
  std::vector<int64_t> e_row0, e_rows, e_zrow0;
  int64_t z_total = 0, max_rows = 0;
  int max_item_rows = 1;
  int tail = 0;                         // fused tail of the gradient kernel
  // tensor-core softmax path: partitions' Z / R rows padded to 64
  std::vector<int64_t> e_zrow0p;
  std::vector<int32_t> f_prefix, f_nk, f_aoff, f_mvalid, b_nk, b_aoff, b_boff;
  // f_mvalid: row tiles of each batch (unfused logits GEMM); b_*: K blocks,
  // R and X row offsets of each batch (gradient contraction)
  std::vector<int64_t> f_outrow0;
  int64_t zpad_total = 0;
  int64_t* d_e_zrow0p = nullptr;
  int32_t *d_f_prefix = nullptr, *d_f_nk = nullptr, *d_f_aoff = nullptr, *d_f_mvalid = nullptr;
  int32_t *d_b_nk = nullptr, *d_b_aoff = nullptr, *d_b_boff = nullptr;
  int64_t* d_f_outrow0 = nullptr;
  // fused logits + residual kernel: 128-row tiles {X row, R row, valid rows, e}
  std::vector<int32_t> q_tiles;
  int32_t* d_q_tiles = nullptr;
  // gradient contraction: units {class pair tile, feature tile, first e, run length}
  std::vector<int32_t> g_units;
  int32_t* d_g_units = nullptr;
  // few-class softmax: 128-row tiles {row0, rows, item, flags} and items
  std::vector<int32_t> sk_tiles;
  int sk_items = 0;
  int32_t* d_sk_tiles = nullptr;
  std::vector<int32_t> sk_cuts;   // whole-row variant: tile range of each CTA pair
  int32_t* d_sk_cuts = nullptr;
  // device copies
  WorkItem* d_items = nullptr;
  int32_t* d_e_item0 = nullptr;
  float* d_e_scale = nullptr;
  int32_t* d_e_dest = nullptr;
  int64_t* d_e_row0 = nullptr;
  int64_t* d_e_rows = nullptr;
  int64_t* d_e_zrow0 = nullptr;
};

bool valid_scheme(int32_t v) { return v == PGC_FR || v == PGC_CR; }
bool valid_loss(int32_t v) { return v == PGC_LOGISTIC || v == PGC_LSQ || v == PGC_SOFTMAX; }
bool valid_dtype(int32_t v) { return v == PGC_F32 || v == PGC_BF16; }

int check_nsc(int32_t scheme, int32_t n, int32_t s) {
  if (!valid_scheme(scheme)) return PGC_EINVAL;
  if (n < 1 || n > kMaxWorkers || s < 0 || s + 1 > n) return PGC_EINVAL;
  if (scheme == PGC_FR && n % (s + 1) != 0) return PGC_EINVAL;
  return PGC_OK;
}

// Partition in slot l of worker i: FR D_{floor(i/c) c + l} (§IV-A),
// CR D_{(i + l) mod n} (§V-B).
inline int32_t held(int32_t scheme, int32_t n, int32_t c, int32_t i, int32_t l) {
  return scheme == PGC_FR ? (i / c) * c + l : (i + l) % n;
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

}  // namespace

struct pgc_ctx {
  int32_t n = 0, s = 0, c = 1, scheme = 0, loss = 0, dtype = 0;
  int64_t d = 0, K = 1, ld = 0, P = 0, Kpad = 0;
  std::vector<int64_t> rows, row0;
  int64_t total_rows = 0;
  float lr = 0.f;
  cudaStream_t stream = nullptr;
  int device = 0, sm_count = 148;
  int variant = -1;          // K1 variant (logistic / least squares)
  int owners = 0;
  size_t esize = 4;

  void* X = nullptr;
  void* y = nullptr;
  float* w = nullptr;
  uint16_t* wb = nullptr;
  float* store = nullptr;
  float* U = nullptr;
  float* gout = nullptr;
  float* partials = nullptr;
  float* Z = nullptr;
  float* coeff = nullptr;
  int* status = nullptr;
  double* loss_blocks = nullptr;
  double* loss_out = nullptr;
  int64_t* loss_desc = nullptr;
  int* counters = nullptr;   // [n + 3]: per-partition arrivals, committed partitions,
                             // work-item counter, finished producers (zero between steps)
  bool pdl = true;           // chain the step's kernels with programmatic dependent launch
  int tail_mode = 0;         // fused tail of the gradient kernel (see GradRowsArgs)
  int mode = PGC_MODE_PGC;   // training scheme (PGC_MODE_*)
  int64_t prefetch_bytes = 0;  // streaming kernel's L2 warm-up per CTA (PGC_PREFETCH_KB)
  bool tc = false;           // softmax on the tensor cores (bf16 features)
  bool smallk = false;       // few-class softmax: one-pass cluster kernel
  int sk_nper = 0;           // its 64-feature blocks per CTA slice
  int sk_nc = 0;             // its clusters (whole-row variant: its CTAs, two per pair)
  bool sk_rows = false;      // the whole-row variant (CTA pairs, kRowsTileRows-row tiles)
  int sk_slots = 0;          // its tile slots
  int sk_box = 1;            // its 64-feature blocks per TMA copy
  bool sk_tail = true;       // its fused commit + decode (PGC_NO_ROWS_TAIL=1: separate kernels)
  alignas(64) unsigned char tmXr[128];   // X as [ld/64][rows][64] blocks (box 64 x kRowsTileRows x sk_box)
  alignas(64) unsigned char tmW16[128];  // Wb [16][ld] for the few-class kernel (box 64 x 16)
  int64_t Ktc = 0;           // classes padded to the forward N tile (256)
  uint16_t* Rb = nullptr;    // bf16 residuals [zpad rows][Ktc]
  float* pre = nullptr;      // fused tensor-core path: the decode's early terms [P]
  int* status_h = nullptr;   // pinned host copy of the status word
  alignas(64) unsigned char tmXk[128];   // X as K-major A   (box 64 x 128)
  alignas(64) unsigned char tmW[128];    // Wb as K-major B  (box 64 x 128: one CTA's half of a 256 tile)
  alignas(64) unsigned char tmR[128];    // R as MN-major A  (box 64 x 64)
  alignas(64) unsigned char tmXm[128];   // X as MN-major B  (box 64 x 64)
  alignas(64) unsigned char tmZo[128];   // Z fp32 output     (box 32 x 32)
  alignas(64) unsigned char tmUo[128];   // U [c][K][ld] fp32, reduce-add target
  alignas(64) unsigned char tmSo[128];   // stores [owners c][K][ld] fp32, TMA store target
  bool tcf = false;          // logits GEMM with the residual fused (no Z in HBM)
  int tcf_nc = 0;            // its clusters of Ktc / 256 CTAs
  int tcg_pairs = 0;         // co-resident CTA pairs of the gradient contraction
  alignas(64) unsigned char tmXq[128];   // X as the fused kernel's A part (box 64 x 128/NT)
  alignas(64) unsigned char tmRst[128];  // Rb as the fused kernel's output (box 64 x 32)
  // GC-CR coding: the naive PGC-CR mode and GC with cyclic repetition (§V-A)
  bool gc_weighted = false;    // decode with GC-CR's weights instead of PGC's slot totals
  bool gc_ready = false;       // encoding coefficients set (pgc_set_gc_encoding)
  double* gc_coeff = nullptr;  // [n][c] encoding coefficients c_{j,l}
  double* gc_d = nullptr;      // [n + 2] the last step's d_j, then max and min alpha
  double* gc_draws = nullptr;  // [s][n-1] the construction's draws (staging)
  float* gc_wts = nullptr;     // [n][c] the last step's d_j c_{j,l} / n
  int64_t loss_chunk = 0;
  int loss_nblocks = 256;
  void* tables = nullptr;

  std::vector<Phase> phases;
  // measurement: events around the kernel groups of each recorded step
  bool timing = false;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  int64_t launches[PGC_NKGROUPS] = {0, 0, 0};
  int64_t timed_steps = 0;
  bool loaded = false;
  bool broken = false;
  bool stepped = false;
  int64_t t = 0;
};

namespace {

thread_local cudaError_t g_last_cuda_error = cudaSuccess;

int cuda_fail(pgc_ctx* ctx, cudaError_t e) {
  if (e == cudaSuccess) return PGC_OK;
  g_last_cuda_error = e;
  if (ctx) ctx->broken = true;
  return e == cudaErrorMemoryAllocation ? PGC_ENOMEM : PGC_ECUDA;
}

#define PGC_CK(ctx, expr)                          \
  do {                                             \
    cudaError_t _e = (expr);                       \
    if (_e != cudaSuccess) return cuda_fail(ctx, _e); \
  } while (0)

// Read and clear nothing: map the device status word to a code.
int read_status(pgc_ctx* ctx) {
  // into pinned memory: the copy is a plain asynchronous one, no staging
  cudaError_t e = cudaMemcpyAsync(ctx->status_h, ctx->status, sizeof(int), cudaMemcpyDeviceToHost, ctx->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e);
  const int h = *ctx->status_h;
  if (h & kErrWaitTimeout) { ctx->broken = true; return PGC_ETIMEOUT; }
  if (h & kErrBadMask) { ctx->broken = true; return PGC_EMASK; }
  if (h & kErrSingular) { ctx->broken = true; return PGC_ESINGULAR; }
  if (h) { ctx->broken = true; return PGC_ECUDA; }
  return PGC_OK;
}

void build_phase(pgc_ctx* ctx, Phase& ph, int slot) {
  const int n = ctx->n, c = ctx->c;
  ph.slot = slot;
  ph.parts.clear();
  if (slot < 0 || ctx->scheme == PGC_CR) {
    for (int k = 0; k < n; ++k) ph.parts.push_back(k);
  } else {
    for (int g = 0; g < n / c; ++g) ph.parts.push_back(g * c + slot);
  }
  const int nE = (int)ph.parts.size();
  // destinations of each new gradient
  if (slot < 0 && ctx->scheme == PGC_CR) {
    ph.ndest = c;
    for (int e = 0; e < nE; ++e) {
      const int k = ph.parts[e];
      for (int l = 0; l < c; ++l) ph.e_dest.push_back(((k - l + n) % n) * c + l);
    }
  } else {
    ph.ndest = 1;
    for (int e = 0; e < nE; ++e) {
      const int k = ph.parts[e];
      if (ctx->scheme == PGC_FR) ph.e_dest.push_back((k / c) * c + (k % c));
      else ph.e_dest.push_back(((k - slot + n) % n) * c + slot);
    }
  }
  int64_t R = 0;
  for (int e = 0; e < nE; ++e) {
    const int k = ph.parts[e];
    ph.e_scale.push_back(1.0f / (float)ctx->rows[k]);
    ph.e_row0.push_back(ctx->row0[k]);
    ph.e_rows.push_back(ctx->rows[k]);
    ph.e_zrow0.push_back(R);
    R += ctx->rows[k];
    ph.max_rows = std::max(ph.max_rows, ctx->rows[k]);
  }
  ph.z_total = R;
  if (ctx->loss != PGC_SOFTMAX) {
    // work items per SM (default 1: one balanced static item per CTA; more are
    // taken dynamically by the persistent grid);
    // an item holds at least one stage of rows.  PGC_ITEMS_PER_SM overrides.
    int per_sm = 1;
    if (const char* env = std::getenv("PGC_ITEMS_PER_SM")) per_sm = std::max(1, std::atoi(env));
    const int64_t G = (int64_t)ctx->sm_count * per_sm;
    const int64_t min_rows = grad_rows_stage_rows(ctx->variant, ctx->ld, ctx->dtype);
    // items of (nearly) one length L for every partition: the smallest L whose
    // item count fits one wave of the grid, so that all CTAs finish together
    // (items of unequal length leave the long ones to fewer CTAs at the end)
    std::vector<int64_t> qe(nE), cap(nE);
    int64_t mmax = 1;
    for (int e = 0; e < nE; ++e) {
      cap[e] = std::max<int64_t>(1, ph.e_rows[e] / min_rows);
      mmax = std::max(mmax, ph.e_rows[e]);
    }
    auto count = [&](int64_t L) {
      int64_t tot = 0;
      for (int e = 0; e < nE; ++e) tot += std::min(cap[e], std::max<int64_t>(1, (ph.e_rows[e] + L - 1) / L));
      return tot;
    };
    int64_t lo = 1, hi = mmax;                 // count(mmax) = nE: the fewest items possible
    while (lo < hi) {
      const int64_t mid = lo + (hi - lo) / 2;
      if (count(mid) <= G) hi = mid; else lo = mid + 1;
    }
    for (int e = 0; e < nE; ++e) qe[e] = std::min(cap[e], std::max<int64_t>(1, (ph.e_rows[e] + lo - 1) / lo));
    ph.e_item0.push_back(0);
    for (int e = 0; e < nE; ++e) {
      const int64_t m = ph.e_rows[e];
      const int64_t q = qe[e];
      for (int64_t i = 0; i < q; ++i) {
        const int64_t a = m * i / q, b = m * (i + 1) / q;
        WorkItem it;
        it.e = e;
        it.part = ph.parts[e];
        it.row0 = ph.e_row0[e] + a;
        it.rows = b - a;
        ph.items.push_back(it);
        ph.max_item_rows = std::max<int>(ph.max_item_rows, (int)(b - a));
      }
      ph.e_item0.push_back((int32_t)ph.items.size());
    }
  } else if (ctx->smallk) {
    // tiles of tr rows in partition order; cluster (whole-row variant: CTA)
    // c takes [T c / nc, T (c+1) / nc); one item per cluster and partition it touches
    const int64_t tr = ctx->sk_rows ? kRowsTileRows : kSmallKRows;
    std::vector<int32_t> te;              // partition of each tile
    for (int e = 0; e < nE; ++e)
      for (int64_t r0 = 0; r0 < ph.e_rows[e]; r0 += tr) {
        ph.sk_tiles.push_back((int32_t)(ph.e_row0[e] + r0));
        ph.sk_tiles.push_back((int32_t)std::min<int64_t>(tr, ph.e_rows[e] - r0));
        ph.sk_tiles.push_back(0);
        ph.sk_tiles.push_back(0);
        te.push_back(e);
      }
    // runs per cluster (whole-row variant: per CTA pair)
    const int64_t T = (int64_t)te.size(), nc = ctx->sk_rows ? ctx->sk_nc / 2 : ctx->sk_nc;
    std::vector<int64_t> cut(nc + 1);
    for (int64_t cl = 0; cl <= nc; ++cl) cut[cl] = T * cl / nc;
    if (ctx->sk_rows) {
      // each tile costs 1 and each run that starts inside a pair's range
      // kRowsDrainTiles more (the previous run's drain stalls the pair); the
      // smallest largest cost whose greedy fill covers every tile
      // (PGC_ROWS_DRAIN_TILES overrides the charge)
      int64_t D = kRowsDrainTiles;
      if (const char* env = std::getenv("PGC_ROWS_DRAIN_TILES")) D = std::max(0, std::atoi(env));
      auto fill = [&](int64_t C) {
        int64_t i = 0;
        for (int64_t p = 0; p < nc; ++p) {
          cut[p] = i;
          int64_t cost = 0;
          while (i < T) {
            const int64_t add = 1 + ((i > cut[p] && te[i] != te[i - 1]) ? D : 0);
            if (cost + add > C) break;
            cost += add;
            ++i;
          }
        }
        cut[nc] = i;
        return i;
      };
      int64_t lo = (T + nc - 1) / nc, hi = lo + D * nE + 1;
      while (lo < hi) {
        const int64_t mid = lo + (hi - lo) / 2;
        if (fill(mid) >= T) hi = mid; else lo = mid + 1;
      }
      fill(lo);
      for (int64_t cl = 0; cl <= nc; ++cl) ph.sk_cuts.push_back((int32_t)cut[cl]);
    }
    std::vector<int32_t> items_of(nE, 0);
    int item = 0;
    for (int64_t cl = 0; cl < nc; ++cl) {
      const int64_t a = cut[cl], b = cut[cl + 1];
      for (int64_t i = a; i < b; ++i) {
        const bool first = i == a || te[i] != te[i - 1];
        const bool last = i == b - 1 || te[i] != te[i + 1];
        if (first) { ++items_of[te[i]]; ++item; }
        ph.sk_tiles[4 * i + 2] = item - 1;
        ph.sk_tiles[4 * i + 3] = (first ? 1 : 0) | (last ? 2 : 0);
      }
    }
    ph.sk_items = item;
    ph.e_item0.push_back(0);
    for (int e = 0; e < nE; ++e) ph.e_item0.push_back(ph.e_item0.back() + items_of[e]);
  } else {
    for (int e = 0; e <= nE; ++e) ph.e_item0.push_back(e);
    if (ctx->tc) {
      const int NTf = (int)(ctx->Ktc / 256), MTb = (int)(ctx->Ktc / 128), NTb = (int)(ctx->ld / 256);
      int64_t zp = 0;
      ph.f_prefix.push_back(0);
      for (int e = 0; e < nE; ++e) {
        const int64_t m = ph.e_rows[e];
        ph.e_zrow0p.push_back(zp);
        for (int64_t r = 0; r < m; r += 128) {
          ph.q_tiles.push_back((int32_t)(ph.e_row0[e] + r));
          ph.q_tiles.push_back((int32_t)(zp + r));
          ph.q_tiles.push_back((int32_t)std::min<int64_t>(128, m - r));
          ph.q_tiles.push_back(e);
        }
        ph.f_nk.push_back((int32_t)(ctx->ld / 64));
        ph.f_aoff.push_back((int32_t)ph.e_row0[e]);
        ph.f_outrow0.push_back(zp);
        const int32_t MTf = (int32_t)((m + 127) / 128);
        ph.f_mvalid.push_back(MTf);
        ph.f_prefix.push_back(ph.f_prefix.back() + (MTf + 1) / 2 * NTf);   // pairs of row tiles
        ph.b_nk.push_back((int32_t)((m + 63) / 64));
        ph.b_aoff.push_back((int32_t)zp);
        ph.b_boff.push_back((int32_t)ph.e_row0[e]);
        zp += (m + 127) / 128 * 128;   // whole forward tiles: their TMA stores stay inside the partition
      }
      ph.zpad_total = zp;
      // gradient units: every (class pair tile, feature tile) for runs of gs
      // consecutive partitions; gs balances the rounds over the CTA pairs
      // (ties go to the longer run: fewer reduce-adds into U) while a run's
      // inputs stay well inside L2
      const int64_t PT = (int64_t)(MTb / 2) * NTb, np = std::max(1, ctx->tcg_pairs);
      const double per_part = (double)ph.max_rows * (double)(ctx->ld + ctx->Ktc) * 2.0;
      int gs = 1;
      int64_t best = INT64_MAX;
      for (int g = 1; g <= kTcGradMaxRun; ++g) {
        if (g > 1 && g * per_part > 48.0 * 1024 * 1024) break;
        const int64_t units = (nE + g - 1) / g * PT;
        const int64_t cost = (units + np - 1) / np * g;
        if (cost <= best) { best = cost; gs = g; }
      }
      if (const char* env = std::getenv("PGC_GRAD_RUN")) gs = std::min(kTcGradMaxRun, std::max(1, std::atoi(env)));
      // feature-tile-major within a run: the class-pair tiles that share an X
      // tile are adjacent, so a run split across two waves of CTA pairs
      // fetches only R tiles again, not X (class-pair-major order read
      // X and R 1.54x; this order 1.16x)
      for (int e0 = 0; e0 < nE; e0 += gs)
        for (int nt = 0; nt < NTb; ++nt)
          for (int mp = 0; mp < MTb / 2; ++mp) {
            ph.g_units.push_back(mp);
            ph.g_units.push_back(nt);
            ph.g_units.push_back(e0);
            ph.g_units.push_back(std::min(gs, nE - e0));
          }
    }
  }
}

template <typename T>
void put(std::vector<uint8_t>& buf, size_t& off, const std::vector<T>& v) {
  off = align_up(off, 16);
  const size_t bytes = v.size() * sizeof(T);
  if (buf.size() < off + bytes) buf.resize(off + bytes);
  if (bytes) std::memcpy(buf.data() + off, v.data(), bytes);
  off += bytes;
}

cudaError_t record_event(pgc_ctx* ctx) {
  if (!ctx->timing) return cudaSuccess;
  if (ctx->ev_used == ctx->ev_pool.size()) {
    cudaEvent_t ev;
    cudaError_t e = cudaEventCreate(&ev);
    if (e != cudaSuccess) return e;
    ctx->ev_pool.push_back(ev);
  }
  return cudaEventRecord(ctx->ev_pool[ctx->ev_used++], ctx->stream);
}

void free_all(pgc_ctx* ctx) {
  for (cudaEvent_t ev : ctx->ev_pool) cudaEventDestroy(ev);
  ctx->ev_pool.clear();
  void* ptrs[] = {ctx->X, ctx->y, ctx->w, ctx->wb, ctx->store, ctx->U, ctx->gout, ctx->partials, ctx->Z,
                  ctx->coeff, ctx->status, ctx->loss_blocks, ctx->loss_out, ctx->tables, ctx->counters, ctx->Rb,
                  ctx->gc_coeff, ctx->gc_d, ctx->gc_draws, ctx->gc_wts, ctx->pre};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  if (ctx->status_h) cudaFreeHost(ctx->status_h);
  ctx->status_h = nullptr;
}

// Device address of a pinned host buffer mapped into the current device's
// address space, or nullptr (pageable memory, or not addressable).
void* mapped_host(const void* p) {
  if (!p) return nullptr;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();   // not a CUDA pointer: clear the error
    return nullptr;
  }
  return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}

int copy_out(pgc_ctx* ctx, float* dst, const float* src, int on_device) {
  // unpad [K][ld] -> [K][d]
  const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
  PGC_CK(ctx, cudaMemcpy2DAsync(dst, ctx->d * sizeof(float), src, ctx->ld * sizeof(float), ctx->d * sizeof(float),
                                ctx->K, kind, ctx->stream));
  return PGC_OK;
}

}  // namespace

extern "C" {

const char* pgc_gradient_path(const pgc_ctx* ctx) {
  if (!ctx) return "";
  if (ctx->loss != PGC_SOFTMAX) return "grad_rows";
  if (ctx->tc) return ctx->tcf ? "tc_fused" : "tc";
  if (ctx->smallk) return ctx->sk_rows ? "softmax_rows" : "softmax_cluster";
  return "softmax_cc";
}

const char* pgc_last_cuda_error(void) {
  return g_last_cuda_error == cudaSuccess ? "" : cudaGetErrorName(g_last_cuda_error);
}

const char* pgc_strerror(int32_t code) {
  switch (code) {
    case PGC_OK: return "ok";
    case PGC_EINVAL: return "invalid argument";
    case PGC_EMASK: return "straggler mask must hold exactly s ones and n-s zeros";
    case PGC_ESTATE: return "call out of order (partitions not loaded?)";
    case PGC_ENOMEM: return "out of memory";
    case PGC_ECUDA: return "CUDA error";
    case PGC_ENOTSUP: return "unsupported combination";
    case PGC_ETIMEOUT: return "a bounded device-side wait timed out";
    case PGC_ESCRATCH: return "problem too large for the fixed scratch of pgc_gradient_noalloc";
    case PGC_ESINGULAR: return "GC-CR: singular encoding system, or a straggler set the encoding cannot decode";
    default: return "unknown status";
  }
}

int pgc_placement(int32_t scheme, int32_t n, int32_t s, int32_t* table) {
  const int rc = check_nsc(scheme, n, s);
  if (rc) return rc;
  if (!table) return PGC_EINVAL;
  const int c = s + 1;
  for (int i = 0; i < n; ++i)
    for (int l = 0; l < c; ++l) table[i * c + l] = held(scheme, n, c, i, l);
  return PGC_OK;
}

int pgc_schedule(int32_t scheme, int32_t n, int32_t s, int64_t t, int32_t* eval_partition, int32_t* slot) {
  const int rc = check_nsc(scheme, n, s);
  if (rc) return rc;
  if (t < 0) return PGC_EINVAL;
  const int c = s + 1;
  const int o = t == 0 ? -1 : (int)((t - 1) % c);
  if (slot) *slot = o;
  if (eval_partition)
    for (int i = 0; i < n; ++i) eval_partition[i] = o < 0 ? -1 : held(scheme, n, c, i, o);
  return PGC_OK;
}

int pgc_create(pgc_ctx** out, int32_t n, int32_t s, int32_t scheme, int32_t loss, int32_t dtype, int64_t d,
               int64_t K, const int64_t* rows, float lr, const float* w0, void* stream) {
  return pgc_create_mode(out, PGC_MODE_PGC, n, s, scheme, loss, dtype, d, K, rows, lr, w0, stream);
}

int pgc_create_mode(pgc_ctx** out, int32_t mode, int32_t n, int32_t s, int32_t scheme, int32_t loss,
                    int32_t dtype, int64_t d, int64_t K, const int64_t* rows, float lr, const float* w0,
                    void* stream) {
  if (!out) return PGC_EINVAL;
  *out = nullptr;
  int rc = check_nsc(scheme, n, s);
  if (rc) return rc;
  if (mode != PGC_MODE_PGC && mode != PGC_MODE_IS_SGD && mode != PGC_MODE_GC && mode != PGC_MODE_NAIVE_CR)
    return PGC_EINVAL;
  if ((mode == PGC_MODE_IS_SGD || mode == PGC_MODE_NAIVE_CR) && scheme != PGC_CR) return PGC_EINVAL;
  // GC-CR's decode weights come from per-step fp64 solves on one warp
  const bool gc_weighted = mode == PGC_MODE_NAIVE_CR || (mode == PGC_MODE_GC && scheme == PGC_CR);
  if (gc_weighted && n > kGcMaxN) return PGC_ENOTSUP;
  if (!valid_loss(loss) || !valid_dtype(dtype) || d < 1 || !rows || !std::isfinite(lr)) return PGC_EINVAL;
  if (loss == PGC_SOFTMAX ? (K < 2 || K > 4096) : K != 1) return PGC_EINVAL;
  for (int k = 0; k < n; ++k)
    if (rows[k] < 1) return PGC_EINVAL;
  if (d > (1 << 20)) return PGC_ENOTSUP;

  pgc_ctx* ctx = new (std::nothrow) pgc_ctx();
  if (!ctx) return PGC_ENOMEM;
  // IS-SGD keeps one slot per worker (its own partition) and still ignores s stragglers
  ctx->mode = mode;
  ctx->gc_weighted = gc_weighted;
  ctx->n = n; ctx->s = s; ctx->c = mode == PGC_MODE_IS_SGD ? 1 : s + 1;
  ctx->scheme = scheme; ctx->loss = loss; ctx->dtype = dtype;
  ctx->d = d; ctx->K = K; ctx->lr = lr;
  ctx->stream = static_cast<cudaStream_t>(stream);
  ctx->esize = dtype == PGC_BF16 ? 2 : 4;
  ctx->owners = scheme == PGC_FR ? n / ctx->c : n;
  ctx->rows.assign(rows, rows + n);
  ctx->row0.resize(n);
  int64_t acc = 0;
  for (int k = 0; k < n; ++k) { ctx->row0[k] = acc; acc += rows[k]; }
  ctx->total_rows = acc;

  if (loss != PGC_SOFTMAX) {
    ctx->variant = grad_rows_variant(dtype, d, &ctx->ld);
    if (ctx->variant < 0) { delete ctx; return PGC_ENOTSUP; }
  } else {
    // bf16 softmax runs on the tensor cores (PGC_NO_TC=1 keeps the CUDA-core path)
    const char* env = std::getenv("PGC_NO_TC");
    ctx->tc = dtype == PGC_BF16 && K >= kTcMinClasses && K <= kTcMaxClasses && !(env && env[0] == '1');
    ctx->ld = (int64_t)align_up((size_t)d, ctx->tc ? 256 : 64);
    ctx->Ktc = (int64_t)align_up((size_t)K, 256);
    // the residual runs in the logits GEMM's epilogue when one cluster can
    // hold every class of a row tile (PGC_NO_FUSED=1 keeps three kernels)
    const char* env3 = std::getenv("PGC_NO_FUSED");
    if (ctx->tc) ctx->tcg_pairs = tc_grad_max_pairs();
    if (ctx->tc && !(env3 && env3[0] == '1')) {
      ctx->tcf_nc = tc_softmax_max_clusters((int)(ctx->Ktc / 256));
      ctx->tcf = ctx->tcf_nc > 0;
    }
    const char* env2 = std::getenv("PGC_NO_SMALLK");
    const char* env4 = std::getenv("PGC_NO_ROWS");
    if (!ctx->tc && dtype == PGC_BF16 && !(env2 && env2[0] == '1') && !(env4 && env4[0] == '1') && K <= 16) {
      // few classes, rows short enough to hold 16 whole rows per CTA pair
      // and slot: one CTA per SM, a cluster of two per tile (PGC_NO_ROWS=1
      // keeps the 8-CTA cluster kernel)
      const int64_t ldr = (int64_t)align_up((size_t)d, 256);
      const int slots = rows_slots(ldr);
      // TMA copies of up to 8 blocks (16 KB); PGC_ROWS_BOX requests another count
      int req = 0;
      if (const char* env = std::getenv("PGC_ROWS_BOX")) req = std::atoi(env);
      const int box = rows_box_blocks(ldr, req);
      ctx->sk_box = box;
      if (const char* env = std::getenv("PGC_NO_ROWS_TAIL")) ctx->sk_tail = env[0] != '1';
      if (gc_weighted) ctx->sk_tail = false;   // its fused decode is PGC's
      // the occupancy query first: it makes the runtime's context current,
      // which the tensor-map encoder (a driver call) needs
      const int nctas = slots >= 2 ? rows_max_ctas(ldr, slots) : 0;
      if (nctas > 0 && make_tmap_bf16_rows(nullptr, nullptr, (uint64_t)ldr, 1024, kRowsTileRows, (uint32_t)box)) {
        {
          ctx->ld = ldr;
          ctx->sk_rows = ctx->smallk = true;
          ctx->sk_slots = slots;
          ctx->sk_nc = nctas;
        }
      }
    }
    if (!ctx->tc && !ctx->smallk && dtype == PGC_BF16 && !(env2 && env2[0] == '1') && smallk_fits(K, ctx->ld)) {
      ctx->sk_nper = (int)((ctx->ld / 64 + 7) / 8);
      ctx->sk_nc = smallk_max_clusters(ctx->sk_nper);
      ctx->smallk = ctx->sk_nc > 0;
    }
  }
  ctx->P = ctx->K * ctx->ld;
  ctx->Kpad = (int64_t)align_up((size_t)K, 4);
  if (const char* env = std::getenv("PGC_PREFETCH_KB")) ctx->prefetch_bytes = (int64_t)std::atoll(env) * 1024;
  {
    const char* env = std::getenv("PGC_NO_PDL");
    ctx->pdl = !(env && env[0] == '1');
  }
  if (loss != PGC_SOFTMAX) {
    // fuse the decode into the gradient kernel when one CTA can read what it
    // needs quickly: the refreshed slot of every store, the other slot
    // totals and the stragglers' stores, about (owners + c + s c) P floats
    const double dec_bytes = (double)(ctx->owners + ctx->c + (double)s * ctx->c) * ctx->P * 4.0;
    ctx->tail_mode = dec_bytes <= 512.0 * 1024.0 && !gc_weighted ? 2 : 1;
  }

  cudaError_t e = cudaGetDevice(&ctx->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->sm_count, cudaDevAttrMultiProcessorCount, ctx->device);
  if (e != cudaSuccess) { delete ctx; return PGC_ECUDA; }

  // phases and their tables
  ctx->phases.resize(1 + ctx->c);
  build_phase(ctx, ctx->phases[0], -1);
  for (int o = 0; o < ctx->c; ++o) build_phase(ctx, ctx->phases[1 + o], o);
  for (auto& ph : ctx->phases) ph.tail = ctx->loss == PGC_SOFTMAX ? 0 : ctx->tail_mode;
  size_t max_partials = 0;
  int64_t max_z = 0;
  for (auto& ph : ctx->phases) {
    // the tensor-core backward writes the stores directly: no partials
    const size_t np = ctx->tc ? 0
                      : ctx->smallk ? (size_t)ph.sk_items * ctx->P
                      : ctx->loss == PGC_SOFTMAX ? ph.parts.size() * (size_t)ctx->P
                                                 : ph.items.size() * (size_t)ctx->ld;
    max_partials = std::max(max_partials, np);
    max_z = std::max(max_z, ph.z_total);
  }
  std::vector<uint8_t> tab;
  size_t off = 0;
  std::vector<size_t> offs;
  constexpr int kTabs = 20;
  for (auto& ph : ctx->phases) {
    offs.push_back(align_up(off, 16)); put(tab, off, ph.items);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_item0);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_scale);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_dest);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_row0);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_rows);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_zrow0);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.e_zrow0p);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.f_prefix);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.f_nk);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.f_aoff);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.f_mvalid);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.f_outrow0);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.b_nk);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.b_aoff);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.b_boff);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.sk_tiles);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.q_tiles);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.g_units);
    offs.push_back(align_up(off, 16)); put(tab, off, ph.sk_cuts);
  }
  // loss chunks (softmax): {row0, rows, 0} per chunk
  std::vector<int64_t> ldesc;
  if (loss == PGC_SOFTMAX) {
    ctx->loss_chunk = std::min<int64_t>(ctx->total_rows, 32768);
    for (int64_t r0 = 0; r0 < ctx->total_rows; r0 += ctx->loss_chunk) {
      ldesc.push_back(r0);
      ldesc.push_back(std::min(ctx->loss_chunk, ctx->total_rows - r0));
      ldesc.push_back(0);
    }
  }
  const size_t ldesc_off = align_up(off, 16);
  put(tab, off, ldesc);
  if (tab.empty()) tab.resize(16);

  auto fail = [&](cudaError_t err) {
    free_all(ctx);
    delete ctx;
    return err == cudaErrorMemoryAllocation ? PGC_ENOMEM : PGC_ECUDA;
  };
#define PGC_ALLOC(ptr, bytes)                                              \
  do {                                                                     \
    cudaError_t _e = cudaMalloc((void**)&(ptr), std::max<size_t>((bytes), 16)); \
    if (_e != cudaSuccess) return fail(_e);                                \
  } while (0)

  const size_t Pb = (size_t)ctx->P * sizeof(float);
  PGC_ALLOC(ctx->X, (size_t)ctx->total_rows * ctx->ld * ctx->esize);
  PGC_ALLOC(ctx->y, (size_t)ctx->total_rows * 4 + 64);   // per-stage label copies overrun by <= 12 B
  PGC_ALLOC(ctx->w, Pb);
  const size_t wb_elems = ctx->tc ? (size_t)ctx->Ktc * ctx->ld : ctx->smallk ? (size_t)16 * ctx->ld : (size_t)ctx->P;
  if (dtype == PGC_BF16) PGC_ALLOC(ctx->wb, wb_elems * 2);
  PGC_ALLOC(ctx->store, (size_t)ctx->owners * ctx->c * Pb);
  PGC_ALLOC(ctx->U, (size_t)ctx->c * Pb);
  PGC_ALLOC(ctx->gout, Pb);
  PGC_ALLOC(ctx->partials, max_partials * sizeof(float));
  int64_t max_zpad = 0;
  for (auto& ph : ctx->phases) max_zpad = std::max(max_zpad, ph.zpad_total);
  if (loss == PGC_SOFTMAX) {
    const size_t zcc = (size_t)std::max<int64_t>(max_z, ctx->loss_chunk) * ctx->Kpad;
    const size_t ztc = ctx->tc && !ctx->tcf ? (size_t)max_zpad * ctx->Ktc : 0;
    PGC_ALLOC(ctx->Z, std::max(zcc, ztc) * sizeof(float));
  }
  if (ctx->tc) PGC_ALLOC(ctx->Rb, (size_t)max_zpad * ctx->Ktc * sizeof(uint16_t));
  // The decode's terms of the slots other than o_t are summed by four warps
  // of the fused logits kernel when that pays: the decode after the gradient
  // contraction then reads (c - 1)(1 + s) P floats less (at about 6.5 TB/s),
  // while the warps stream them at about 2.2 TB/s beside a GEMM running at
  // about 1.43 PFLOP/s that gives up about 6 % to them and waits for them if
  // it finishes first.  PGC_PRE_DECODE=1 (=0) forces the split on (off).
  if (ctx->tc && ctx->tcf && !gc_weighted && ctx->P / 4 >= kPreDecodeMinP4 && s <= kPreMaxDev) {
    const int cc = ctx->c;
    const double rows_eval = scheme == PGC_CR ? (double)ctx->total_rows : (double)ctx->total_rows / cc;
    const double pre_bytes = (double)(cc - 1) * (1 + (scheme == PGC_CR ? s : 0)) * (double)ctx->P * 4.0;
    const double t_gemm = 2.0 * rows_eval * (double)ctx->ld * (double)ctx->Ktc / 1.43e15;
    const double t_pre = pre_bytes / 2.2e12;
    const double gain = pre_bytes / 6.5e12 - std::max(0.0, t_pre - t_gemm) - 0.06 * t_gemm;
    bool on = gain > 0.0;
    if (const char* e = std::getenv("PGC_PRE_DECODE")) on = e[0] == '1';
    if (on) PGC_ALLOC(ctx->pre, Pb);
  }
  PGC_ALLOC(ctx->coeff, (size_t)n * sizeof(float));
  PGC_ALLOC(ctx->status, sizeof(int));
  {
    cudaError_t _e = cudaMallocHost((void**)&ctx->status_h, sizeof(int));
    if (_e != cudaSuccess) return fail(_e);
  }
  PGC_ALLOC(ctx->loss_blocks, (size_t)ctx->loss_nblocks * sizeof(double));
  PGC_ALLOC(ctx->loss_out, sizeof(double));
  PGC_ALLOC(ctx->tables, tab.size());
  PGC_ALLOC(ctx->counters, (size_t)(n + 3) * sizeof(int));
  if (gc_weighted) {
    PGC_ALLOC(ctx->gc_coeff, (size_t)n * ctx->c * sizeof(double));
    PGC_ALLOC(ctx->gc_d, (size_t)(n + 2) * sizeof(double));
    PGC_ALLOC(ctx->gc_draws, (size_t)s * (n - 1) * sizeof(double));
    PGC_ALLOC(ctx->gc_wts, (size_t)n * ctx->c * sizeof(float));
  }

  cudaStream_t st = ctx->stream;
  e = cudaMemcpyAsync(ctx->tables, tab.data(), tab.size(), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->X, 0, (size_t)ctx->total_rows * ctx->ld * ctx->esize, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->w, 0, Pb, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->store, 0, (size_t)ctx->owners * ctx->c * Pb, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->U, 0, (size_t)ctx->c * Pb, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->gout, 0, Pb, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->coeff, 0, (size_t)n * sizeof(float), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->status, 0, sizeof(int), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->counters, 0, (size_t)(n + 3) * sizeof(int), st);
  if (e == cudaSuccess && gc_weighted) e = cudaMemsetAsync(ctx->gc_wts, 0, (size_t)n * ctx->c * sizeof(float), st);
  if (e == cudaSuccess && gc_weighted) e = cudaMemsetAsync(ctx->gc_d, 0, (size_t)(n + 2) * sizeof(double), st);
  if (e == cudaSuccess && w0)
    e = cudaMemcpy2DAsync(ctx->w, ctx->ld * sizeof(float), w0, d * sizeof(float), d * sizeof(float), K,
                          cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && ctx->wb) e = cudaMemsetAsync(ctx->wb, 0, wb_elems * 2, st);
  if (e == cudaSuccess && ctx->wb) e = launch_f32_to_bf16(ctx->w, ctx->wb, ctx->P, st);
  if (e == cudaSuccess && ctx->Rb) e = cudaMemsetAsync(ctx->Rb, 0, (size_t)max_zpad * ctx->Ktc * 2, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail(e);

  uint8_t* base = static_cast<uint8_t*>(ctx->tables);
  for (size_t i = 0; i < ctx->phases.size(); ++i) {
    Phase& ph = ctx->phases[i];
    const size_t* o = &offs[kTabs * i];
    ph.d_items = reinterpret_cast<WorkItem*>(base + o[0]);
    ph.d_e_item0 = reinterpret_cast<int32_t*>(base + o[1]);
    ph.d_e_scale = reinterpret_cast<float*>(base + o[2]);
    ph.d_e_dest = reinterpret_cast<int32_t*>(base + o[3]);
    ph.d_e_row0 = reinterpret_cast<int64_t*>(base + o[4]);
    ph.d_e_rows = reinterpret_cast<int64_t*>(base + o[5]);
    ph.d_e_zrow0 = reinterpret_cast<int64_t*>(base + o[6]);
    ph.d_e_zrow0p = reinterpret_cast<int64_t*>(base + o[7]);
    ph.d_f_prefix = reinterpret_cast<int32_t*>(base + o[8]);
    ph.d_f_nk = reinterpret_cast<int32_t*>(base + o[9]);
    ph.d_f_aoff = reinterpret_cast<int32_t*>(base + o[10]);
    ph.d_f_mvalid = reinterpret_cast<int32_t*>(base + o[11]);
    ph.d_f_outrow0 = reinterpret_cast<int64_t*>(base + o[12]);
    ph.d_b_nk = reinterpret_cast<int32_t*>(base + o[13]);
    ph.d_b_aoff = reinterpret_cast<int32_t*>(base + o[14]);
    ph.d_b_boff = reinterpret_cast<int32_t*>(base + o[15]);
    ph.d_sk_tiles = reinterpret_cast<int32_t*>(base + o[16]);
    ph.d_q_tiles = reinterpret_cast<int32_t*>(base + o[17]);
    ph.d_g_units = reinterpret_cast<int32_t*>(base + o[18]);
    ph.d_sk_cuts = reinterpret_cast<int32_t*>(base + o[19]);
  }
  ctx->loss_desc = nullptr;
  if (!ldesc.empty()) ctx->loss_desc = reinterpret_cast<int64_t*>(base + ldesc_off);
  if (ctx->sk_rows) {
    if (!make_tmap_bf16_rows(ctx->tmXr, ctx->X, (uint64_t)ctx->ld, (uint64_t)ctx->total_rows, kRowsTileRows,
                             (uint32_t)ctx->sk_box))
      return fail(cudaErrorInvalidValue);
  } else if (ctx->smallk) {
    const uint64_t pitch = (uint64_t)ctx->ld * 2;
    if (!make_tmap_bf16(ctx->tmXk, ctx->X, ctx->ld, ctx->total_rows, pitch, kSmallKRows) ||
        !make_tmap_bf16(ctx->tmW16, ctx->wb, ctx->ld, 16, pitch, 16))
      return fail(cudaErrorInvalidValue);
  }
  if (ctx->tc) {
    const uint64_t pitch = (uint64_t)ctx->ld * 2;
    bool ok = make_tmap_bf16(ctx->tmXk, ctx->X, ctx->ld, ctx->total_rows, pitch, 128) &&
              make_tmap_bf16(ctx->tmW, ctx->wb, ctx->ld, ctx->Ktc, pitch, 128) &&
              make_tmap_bf16(ctx->tmR, ctx->Rb, ctx->Ktc, max_zpad, (uint64_t)ctx->Ktc * 2, 64) &&
              make_tmap_bf16(ctx->tmXm, ctx->X, ctx->ld, ctx->total_rows, pitch, 64);
    const uint64_t zd[2] = {(uint64_t)ctx->Ktc, (uint64_t)max_zpad}, zs[1] = {(uint64_t)ctx->Ktc * 4};
    const uint64_t ud[3] = {(uint64_t)ctx->ld, (uint64_t)ctx->K, (uint64_t)ctx->c};
    const uint64_t ss[2] = {(uint64_t)ctx->ld * 4, (uint64_t)ctx->P * 4};
    const uint64_t sd[3] = {(uint64_t)ctx->ld, (uint64_t)ctx->K, (uint64_t)ctx->owners * ctx->c};
    ok = ok && make_tmap_f32_box32(ctx->tmUo, ctx->U, 3, ud, ss) && make_tmap_f32_box32(ctx->tmSo, ctx->store, 3, sd, ss);
    if (ctx->tcf)
      ok = ok && make_tmap_bf16(ctx->tmXq, ctx->X, ctx->ld, ctx->total_rows, pitch, (uint32_t)(128 / (ctx->Ktc / 256))) &&
           make_tmap_bf16(ctx->tmRst, ctx->Rb, ctx->Ktc, max_zpad, (uint64_t)ctx->Ktc * 2, 32);
    else
      ok = ok && make_tmap_f32_box32(ctx->tmZo, ctx->Z, 2, zd, zs);
    if (!ok) return fail(cudaErrorInvalidValue);
  }
#undef PGC_ALLOC
  *out = ctx;
  return PGC_OK;
}

int pgc_destroy(pgc_ctx* ctx) {
  if (!ctx) return PGC_OK;
  cudaStreamSynchronize(ctx->stream);
  // loss_desc points into tables; do not free it twice
  ctx->loss_desc = nullptr;
  free_all(ctx);
  delete ctx;
  return PGC_OK;
}

int pgc_load_partitions(pgc_ctx* ctx, const void* const* X, const void* const* y, int32_t on_device) {
  if (!ctx || !X || !y) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  for (int k = 0; k < ctx->n; ++k)
    if (!X[k] || !y[k]) return PGC_EINVAL;
  const cudaMemcpyKind kx = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  const size_t es = ctx->esize;
  for (int k = 0; k < ctx->n; ++k) {
    uint8_t* dst = static_cast<uint8_t*>(ctx->X) + (size_t)ctx->row0[k] * ctx->ld * es;
    PGC_CK(ctx, cudaMemcpy2DAsync(dst, ctx->ld * es, X[k], ctx->d * es, ctx->d * es, ctx->rows[k], kx, ctx->stream));
    PGC_CK(ctx, cudaMemcpyAsync(static_cast<uint8_t*>(ctx->y) + (size_t)ctx->row0[k] * 4, y[k],
                                (size_t)ctx->rows[k] * 4, kx, ctx->stream));
  }
  PGC_CK(ctx, cudaStreamSynchronize(ctx->stream));
  ctx->loaded = true;
  return PGC_OK;
}

int pgc_step(pgc_ctx* ctx, const uint8_t* mask, float* grad_out, float* w_out, int32_t outputs_on_device,
             pgc_step_info* info) {
  if (!ctx || !mask) return PGC_EINVAL;
  if (!ctx->loaded || ctx->broken) return PGC_ESTATE;
  if (ctx->gc_weighted && !ctx->gc_ready) return PGC_ESTATE;
  const int n = ctx->n, c = ctx->c;
  MaskBits bits;
  std::memset(&bits, 0, sizeof(bits));
  int cnt = 0;
  for (int i = 0; i < n; ++i) {
    if (mask[i] > 1) return PGC_EMASK;
    if (mask[i]) { bits.w[i >> 5] |= 1u << (i & 31); ++cnt; }
  }
  if (cnt != ctx->s) return PGC_EMASK;

  const int64_t t = ctx->t;
  // GC refreshes every slot every step (the warm-up phase); IS-SGD's one slot
  // is refreshed every step, t = 0 included
  const int pidx = ctx->mode == PGC_MODE_GC ? 0
                   : ctx->mode == PGC_MODE_IS_SGD ? 1
                   : t == 0 ? 0 : 1 + (int)((t - 1) % c);
  Phase& ph = ctx->phases[pidx];
  cudaStream_t st = ctx->stream;

  PGC_CK(ctx, record_event(ctx));
  int64_t nl[PGC_NKGROUPS] = {0, 0, 0, 0, 0};
  DecodeArgs dc;
  dc.scheme = ctx->scheme; dc.n = n; dc.s = ctx->s; dc.c = c; dc.slot = ph.slot; dc.owners = ctx->owners;
  dc.mask = bits; dc.P = ctx->P; dc.store = ctx->store; dc.U = ctx->U; dc.w = ctx->w; dc.wb = ctx->wb;
  dc.gout = ctx->gout; dc.lr = ctx->lr; dc.coeff_out = ctx->coeff; dc.status = ctx->status;
  // outputs with the unpadded layout (ld == d) and 16-byte alignment that the
  // GPU can address are written by the decode itself: device outputs (so no
  // copy sits between consecutive steps), and pinned host outputs mapped into
  // the device's address space (so no device-to-host copies follow the decode)
  float* g_dev = grad_out;
  float* w_dev = w_out;
  bool direct = ctx->ld == ctx->d && (reinterpret_cast<uintptr_t>(grad_out) % 16 == 0) &&
                (reinterpret_cast<uintptr_t>(w_out) % 16 == 0);
  if (direct && !outputs_on_device) {
    g_dev = static_cast<float*>(mapped_host(grad_out));
    w_dev = static_cast<float*>(mapped_host(w_out));
    direct = (!grad_out || g_dev) && (!w_out || w_dev) && (reinterpret_cast<uintptr_t>(g_dev) % 16 == 0) &&
             (reinterpret_cast<uintptr_t>(w_dev) % 16 == 0);
  }
  if (direct) { dc.g_user = g_dev; dc.w_user = w_dev; }
  bool need_commit = true, need_decode = true;
  if (ctx->loss != PGC_SOFTMAX) {
    // K1 with its fused tail: commit (and, for small P, decode) in the same launch
    GradRowsArgs g;
    g.loss = ctx->loss; g.dtype = ctx->dtype; g.d = ctx->d; g.ld = ctx->ld;
    g.X = ctx->X; g.y = static_cast<const float*>(ctx->y); g.w = ctx->w;
    g.items = ph.d_items; g.nitems = (int)ph.items.size(); g.max_item_rows = ph.max_item_rows;
    g.partials = ctx->partials; g.status = ctx->status;
    g.tail = ph.tail; g.pdl = ctx->pdl;
    g.prefetch_bytes = ctx->prefetch_bytes;
    g.cnt_e = ctx->counters; g.cnt_all = ctx->counters + n;
    g.work_ctr = ctx->counters + n + 1; g.prod_done = ctx->counters + n + 2; g.grid = ctx->sm_count;
    g.e_item0 = ph.d_e_item0; g.e_scale = ph.d_e_scale; g.e_dest = ph.d_e_dest; g.ndest = ph.ndest;
    g.nE = (int)ph.parts.size(); g.store = ctx->store; g.dec = dc;
    nl[PGC_KGRAD] = 1;
    PGC_CK(ctx, launch_grad_rows(g, ctx->variant, st));
    need_commit = false;
    need_decode = ph.tail < 2;
  } else if (ctx->tc) {
    // tensor cores: Z = X Wb^T, R = softmax(Z) - onehot(y) in bf16, then
    // G_e = (1/m_e) R_e^T X_e written straight into the stores
    const int nE = (int)ph.parts.size();
    TcGemmParams f = {};
    f.nbatch = nE; f.tile_prefix = ph.d_f_prefix; f.mt_count = ph.d_f_mvalid; f.NT = (int)(ctx->Ktc / 256); f.nk = ph.d_f_nk;
    // in steady phases every evaluated partition has one store at slot o_t,
    // so the backward also forms U[o_t] = sum_e g_e (TMA reduce-add) and the
    // decode reads it instead of re-summing the stores
    const bool u_red = ph.slot >= 0 && ph.ndest == 1 && !ctx->gc_weighted;
    f.a_off = ph.d_f_aoff; f.total_tiles = ph.f_prefix.back();
    f.out_row0 = ph.d_f_outrow0; f.status = ctx->status; f.pdl = ctx->pdl ? 1 : 0;
    if (ctx->tcf) {
      // R straight from the logits GEMM's epilogue
      TcSoftmaxParams q = {};
      q.tiles = reinterpret_cast<const int4*>(ph.d_q_tiles); q.ntiles = (int)(ph.q_tiles.size() / 4);
      q.NT = (int)(ctx->Ktc / 256); q.nk = (int)(ctx->ld / 64); q.K = (int)ctx->K;
      q.y = static_cast<const int32_t*>(ctx->y);
      q.zero_buf = u_red ? ctx->U + (size_t)ph.slot * ctx->P : nullptr; q.zero_n4 = ctx->P / 4;
      q.status = ctx->status; q.pdl = ctx->pdl ? 1 : 0;
      if (u_red && ctx->pre) {
        // the decode's terms of the slots other than o_t, summed beside the GEMM
        q.pre = dc;
        q.pre_out = ctx->pre;
        dc.pre = ctx->pre;
      }
      PGC_CK(ctx, launch_tc_softmax(ctx->tmXq, ctx->tmW, ctx->tmRst, q, ctx->tcf_nc, st));
      PGC_CK(ctx, record_event(ctx));
      PGC_CK(ctx, record_event(ctx));   // empty residual group
    } else {
      PGC_CK(ctx, launch_tc_gemm(ctx->tmXk, ctx->tmW, ctx->tmZo, f, ctx->sm_count, st));
      PGC_CK(ctx, record_event(ctx));
      PGC_CK(ctx, launch_softmax_bf16(ctx->Z, ctx->Rb, ctx->Ktc, ctx->K, static_cast<const int32_t*>(ctx->y),
                                      ph.d_e_row0, ph.d_e_rows, ph.d_e_zrow0p, nE, ph.max_rows,
                                      u_red ? ctx->U + (size_t)ph.slot * ctx->P : nullptr, ctx->P, st));
      PGC_CK(ctx, record_event(ctx));
    }
    TcGradParams b = {};
    b.units = reinterpret_cast<const int4*>(ph.d_g_units); b.nunits = (int)(ph.g_units.size() / 4);
    b.nk = ph.d_b_nk; b.a_off = ph.d_b_aoff; b.b_off = ph.d_b_boff;
    b.scale = ph.d_e_scale; b.dest = ph.d_e_dest; b.ndest = ph.ndest; b.m_limit = (int)ctx->K;
    b.u_reduce = u_red ? 1 : 0; b.u_slot = ph.slot;
    b.status = ctx->status; b.pdl = ctx->pdl ? 1 : 0;
    PGC_CK(ctx, launch_tc_grad(ctx->tmR, ctx->tmXm, ctx->tmUo, ctx->tmSo, b, ctx->tcg_pairs, st));
    dc.u_ready = u_red ? 1 : 0;
    nl[PGC_KGRAD] = 1;
    nl[PGC_KRESID] = ctx->tcf ? 0 : 1;
    nl[PGC_KGRADB] = 1;
    need_commit = false;
  } else if (ctx->sk_rows) {
    RowsArgs a;
    a.pair_t0 = ph.d_sk_cuts;
    a.tiles = reinterpret_cast<const int4*>(ph.d_sk_tiles); a.ntiles = (int)(ph.sk_tiles.size() / 4);
    a.K = (int)ctx->K; a.y = static_cast<const int32_t*>(ctx->y); a.wb = ctx->wb;
    a.partials = ctx->partials; a.P = ctx->P; a.ld = ctx->ld; a.nslots = ctx->sk_slots; a.box_blocks = ctx->sk_box;
    a.status = ctx->status; a.pdl = ctx->pdl ? 1 : 0;
    if (ctx->sk_tail) {
      // one kernel per step: commit and decode in the same grid
      a.tail = 1; a.nE = (int)ph.parts.size(); a.e_item0 = ph.d_e_item0; a.e_scale = ph.d_e_scale;
      a.e_dest = ph.d_e_dest; a.ndest = ph.ndest; a.store = ctx->store; a.counters = ctx->counters + n;
      a.dec = dc;
      need_commit = false;
      need_decode = false;
    }
    nl[PGC_KGRAD] = 1;
    PGC_CK(ctx, launch_softmax_rows(ctx->tmXr, a, ctx->sk_nc, st));
  } else if (ctx->smallk) {
    SmallKArgs a;
    a.tiles = reinterpret_cast<const int4*>(ph.d_sk_tiles); a.ntiles = (int)(ph.sk_tiles.size() / 4);
    a.nkb = (int)(ctx->ld / 64); a.nper = ctx->sk_nper; a.K = (int)ctx->K;
    a.y = static_cast<const int32_t*>(ctx->y); a.partials = ctx->partials; a.P = ctx->P; a.ld = ctx->ld;
    a.status = ctx->status; a.pdl = ctx->pdl ? 1 : 0;
    nl[PGC_KGRAD] = 1;
    PGC_CK(ctx, launch_softmax_smallk(ctx->tmXk, ctx->tmW16, a, ctx->sk_nc, st));
  } else {
    SoftmaxCCArgs a;
    a.dtype = ctx->dtype; a.ld = ctx->ld; a.K = ctx->K; a.X = ctx->X; a.y = static_cast<const int32_t*>(ctx->y);
    a.W = ctx->w; a.e_row0 = ph.d_e_row0; a.e_rows = ph.d_e_rows; a.e_zrow0 = ph.d_e_zrow0;
    a.nE = (int)ph.parts.size(); a.max_rows = ph.max_rows; a.z_total = ph.z_total; a.Z = ctx->Z;
    a.Kpad = ctx->Kpad; a.partials = ctx->partials;
    nl[PGC_KGRAD] = 3;
    PGC_CK(ctx, launch_softmax_cc(a, st));
  }
  if (!ctx->tc) {
    PGC_CK(ctx, record_event(ctx));   // empty residual and backward groups
    PGC_CK(ctx, record_event(ctx));
  }
  PGC_CK(ctx, record_event(ctx));
  if (need_commit) {
    // K4 commit into the stores
    CommitArgs cm;
    cm.partials = ctx->partials; cm.P = ctx->P; cm.e_item0 = ph.d_e_item0; cm.e_scale = ph.d_e_scale;
    cm.e_dest = ph.d_e_dest; cm.ndest = ph.ndest; cm.nE = (int)ph.parts.size(); cm.store = ctx->store;
    nl[PGC_KCOMMIT] = 1;
    PGC_CK(ctx, launch_commit(cm, st, ctx->pdl));
  }
  PGC_CK(ctx, record_event(ctx));
  if (need_decode && ctx->gc_weighted) {
    // GC-CR: the step's decode weights (one CTA, fp64), then the weighted decode + SGD
    GcWeightsArgs gw;
    gw.n = n; gw.s = ctx->s; gw.c = c; gw.mask = bits; gw.coeff = ctx->gc_coeff; gw.d = ctx->gc_d;
    gw.wts = ctx->gc_wts; gw.coeff_out = ctx->coeff; gw.alpha = ctx->gc_d + n; gw.status = ctx->status;
    nl[PGC_KDECODE] = 2;
    PGC_CK(ctx, launch_gc_decode(gw, dc, st, ctx->pdl, ctx->sm_count));
  } else if (need_decode) {
    // K5+K6 decode + SGD
    nl[PGC_KDECODE] = 1;
    PGC_CK(ctx, launch_decode(dc, st, ctx->pdl, ctx->sm_count));
  }
  PGC_CK(ctx, record_event(ctx));
  if (ctx->timing) {
    for (int k = 0; k < PGC_NKGROUPS; ++k) ctx->launches[k] += nl[k];
    ++ctx->timed_steps;
  }

  if (grad_out && !direct) { int rc = copy_out(ctx, grad_out, ctx->gout, outputs_on_device); if (rc) return rc; }
  if (w_out && !direct) { int rc = copy_out(ctx, w_out, ctx->w, outputs_on_device); if (rc) return rc; }
  if (!outputs_on_device && (grad_out || w_out)) {
    const int rc = read_status(ctx);
    if (rc) return rc;
  }
  if (info) {
    info->t = t;
    info->slot = ph.slot;
    info->received = n - ctx->s;
    if (info->eval_partition)
      for (int i = 0; i < n; ++i) info->eval_partition[i] = ph.slot < 0 ? -1 : held(ctx->scheme, n, c, i, ph.slot);
    if (info->fr_rep && ctx->scheme == PGC_FR)
      for (int g = 0; g < n / c; ++g) {
        int rep = -1;
        for (int l = 0; l < c && rep < 0; ++l)
          if (!mask[g * c + l]) rep = g * c + l;
        info->fr_rep[g] = rep;
      }
  }
  ctx->t = t + 1;
  ctx->stepped = true;
  return PGC_OK;
}

int pgc_sync(pgc_ctx* ctx) {
  if (!ctx) return PGC_EINVAL;
  return read_status(ctx);
}

int pgc_loss(pgc_ctx* ctx, double* loss_out) {
  if (!ctx || !loss_out) return PGC_EINVAL;
  if (!ctx->loaded || ctx->broken) return PGC_ESTATE;
  LossArgs a;
  a.loss = ctx->loss; a.dtype = ctx->dtype; a.ld = ctx->ld; a.K = ctx->K; a.rows = ctx->total_rows;
  a.X = ctx->X; a.y = ctx->y; a.w = ctx->w; a.blocksum = ctx->loss_blocks; a.nblocks = ctx->loss_nblocks;
  a.out = ctx->loss_out; a.Z = ctx->Z; a.Kpad = ctx->Kpad; a.z_chunk_rows = ctx->loss_chunk;
  a.chunk_desc = ctx->loss_desc;
  PGC_CK(ctx, launch_loss(a, ctx->stream));
  PGC_CK(ctx, cudaMemcpyAsync(loss_out, ctx->loss_out, sizeof(double), cudaMemcpyDeviceToHost, ctx->stream));
  return read_status(ctx);
}

int pgc_get_store(pgc_ctx* ctx, int32_t worker, int32_t slot, float* out) {
  if (!ctx || !out || worker < 0 || worker >= ctx->n || slot < 0 || slot >= ctx->c) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  const int owner = ctx->scheme == PGC_FR ? worker / ctx->c : worker;
  const float* src = ctx->store + ((size_t)owner * ctx->c + slot) * ctx->P;
  int rc = copy_out(ctx, out, src, 0);
  if (rc) return rc;
  return read_status(ctx);
}

int pgc_get_store_cols(pgc_ctx* ctx, int32_t worker, int32_t slot, int64_t col0, int64_t ncols, float* out) {
  if (!ctx || !out || worker < 0 || worker >= ctx->n || slot < 0 || slot >= ctx->c) return PGC_EINVAL;
  if (col0 < 0 || ncols < 0 || col0 + ncols > ctx->K * ctx->d) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  const int owner = ctx->scheme == PGC_FR ? worker / ctx->c : worker;
  const float* src = ctx->store + ((size_t)owner * ctx->c + slot) * ctx->P;
  // flattened index k*d + j lives at k*ld + j: one copy per class row touched
  int64_t done = 0;
  while (done < ncols) {
    const int64_t col = col0 + done, k = col / ctx->d, j = col % ctx->d;
    const int64_t len = std::min<int64_t>(ncols - done, ctx->d - j);
    PGC_CK(ctx, cudaMemcpyAsync(out + done, src + k * ctx->ld + j, (size_t)len * sizeof(float),
                                cudaMemcpyDeviceToHost, ctx->stream));
    done += len;
  }
  return read_status(ctx);
}

int pgc_get_decode(pgc_ctx* ctx, float* coeff) {
  if (!ctx || !coeff) return PGC_EINVAL;
  if (!ctx->stepped || ctx->broken) return PGC_ESTATE;
  PGC_CK(ctx, cudaMemcpyAsync(coeff, ctx->coeff, (size_t)ctx->n * sizeof(float), cudaMemcpyDeviceToHost, ctx->stream));
  return read_status(ctx);
}

int pgc_set_gc_encoding(pgc_ctx* ctx, const double* draws) {
  if (!ctx || !ctx->gc_weighted) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  const int n = ctx->n, s = ctx->s;
  if (s > 0 && !draws) return PGC_EINVAL;
  for (int64_t i = 0; i < (int64_t)s * (n - 1); ++i)
    if (!std::isfinite(draws[i])) return PGC_EINVAL;
  cudaStream_t st = ctx->stream;
  if (s > 0)
    PGC_CK(ctx, cudaMemcpyAsync(ctx->gc_draws, draws, (size_t)s * (n - 1) * sizeof(double), cudaMemcpyHostToDevice, st));
  PGC_CK(ctx, launch_gc_encoding(ctx->gc_draws, n, s, ctx->gc_coeff, ctx->status, st));
  int h = 0;
  PGC_CK(ctx, cudaMemcpyAsync(&h, ctx->status, sizeof(int), cudaMemcpyDeviceToHost, st));
  PGC_CK(ctx, cudaStreamSynchronize(st));
  if (h == kErrSingular) {
    // the draws leave some worker's system singular: keep the context usable
    PGC_CK(ctx, cudaMemsetAsync(ctx->status, 0, sizeof(int), st));
    PGC_CK(ctx, cudaStreamSynchronize(st));
    ctx->gc_ready = false;
    return PGC_ESINGULAR;
  }
  if (h) return read_status(ctx);
  ctx->gc_ready = true;
  return PGC_OK;
}

int pgc_get_gc_encoding(pgc_ctx* ctx, double* coeff) {
  if (!ctx || !coeff || !ctx->gc_weighted) return PGC_EINVAL;
  if (!ctx->gc_ready || ctx->broken) return PGC_ESTATE;
  PGC_CK(ctx, cudaMemcpyAsync(coeff, ctx->gc_coeff, (size_t)ctx->n * ctx->c * sizeof(double), cudaMemcpyDeviceToHost,
                              ctx->stream));
  return read_status(ctx);
}

int pgc_get_gc_decode(pgc_ctx* ctx, double* d, double* alpha_range) {
  if (!ctx || !ctx->gc_weighted || (!d && !alpha_range)) return PGC_EINVAL;
  if (!ctx->stepped || ctx->broken) return PGC_ESTATE;
  if (d)
    PGC_CK(ctx, cudaMemcpyAsync(d, ctx->gc_d, (size_t)ctx->n * sizeof(double), cudaMemcpyDeviceToHost, ctx->stream));
  if (alpha_range)
    PGC_CK(ctx, cudaMemcpyAsync(alpha_range, ctx->gc_d + ctx->n, 2 * sizeof(double), cudaMemcpyDeviceToHost,
                                ctx->stream));
  return read_status(ctx);
}

int pgc_get_weights(pgc_ctx* ctx, float* out) {
  if (!ctx || !out) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  int rc = copy_out(ctx, out, ctx->w, 0);
  if (rc) return rc;
  return read_status(ctx);
}

int pgc_set_weights(pgc_ctx* ctx, const float* w) {
  if (!ctx || !w) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  PGC_CK(ctx, cudaMemcpy2DAsync(ctx->w, ctx->ld * sizeof(float), w, ctx->d * sizeof(float), ctx->d * sizeof(float),
                                ctx->K, cudaMemcpyHostToDevice, ctx->stream));
  if (ctx->wb) PGC_CK(ctx, launch_f32_to_bf16(ctx->w, ctx->wb, ctx->P, ctx->stream));
  return read_status(ctx);
}

// ---- checkpoint --------------------------------------------------------------
namespace {
constexpr int64_t kCkptMagic = 0x3154504B43434750LL;   // "PGCCKPT1" little-endian
constexpr int kCkptHeader = 13;
int64_t ckpt_bytes(const pgc_ctx* ctx) {
  const int64_t Kd = ctx->K * ctx->d;
  return kCkptHeader * 8 + 4 * (Kd + (int64_t)ctx->owners * ctx->c * Kd + (int64_t)ctx->c * Kd);
}
void ckpt_header(const pgc_ctx* ctx, int64_t* h) {
  const int64_t v[kCkptHeader] = {kCkptMagic, 1, ctx->mode, ctx->scheme, ctx->loss, ctx->dtype, ctx->n, ctx->s,
                                  ctx->c, ctx->d, ctx->K, ctx->t, ctx->stepped ? 1 : 0};
  for (int i = 0; i < kCkptHeader; ++i) h[i] = v[i];
}
}  // namespace

int pgc_checkpoint_bytes(pgc_ctx* ctx, int64_t* bytes) {
  if (!ctx || !bytes) return PGC_EINVAL;
  *bytes = ckpt_bytes(ctx);
  return PGC_OK;
}

int pgc_checkpoint_save(pgc_ctx* ctx, void* buf, int64_t bytes) {
  if (!ctx || !buf || bytes != ckpt_bytes(ctx)) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  int64_t* h = static_cast<int64_t*>(buf);
  ckpt_header(ctx, h);
  float* p = reinterpret_cast<float*>(h + kCkptHeader);
  const int64_t Kd = ctx->K * ctx->d;
  int rc = copy_out(ctx, p, ctx->w, 0);
  if (rc) return rc;
  p += Kd;
  for (int64_t r = 0; r < (int64_t)ctx->owners * ctx->c; ++r, p += Kd)
    if ((rc = copy_out(ctx, p, ctx->store + r * ctx->P, 0))) return rc;
  for (int o = 0; o < ctx->c; ++o, p += Kd)
    if ((rc = copy_out(ctx, p, ctx->U + (int64_t)o * ctx->P, 0))) return rc;
  return read_status(ctx);
}

int pgc_checkpoint_load(pgc_ctx* ctx, const void* buf, int64_t bytes) {
  if (!ctx || !buf || bytes != ckpt_bytes(ctx)) return PGC_EINVAL;
  if (ctx->broken) return PGC_ESTATE;
  const int64_t* h = static_cast<const int64_t*>(buf);
  int64_t want[kCkptHeader];
  ckpt_header(ctx, want);
  // magic, version and the configuration must match; t and stepped are restored
  for (int i = 0; i < kCkptHeader - 2; ++i)
    if (h[i] != want[i]) return PGC_EINVAL;
  if (h[11] < 0) return PGC_EINVAL;
  const float* p = reinterpret_cast<const float*>(h + kCkptHeader);
  const int64_t Kd = ctx->K * ctx->d;
  auto copy_in = [&](float* dst, const float* src) {
    return cudaMemcpy2DAsync(dst, ctx->ld * sizeof(float), src, ctx->d * sizeof(float), ctx->d * sizeof(float),
                             ctx->K, cudaMemcpyHostToDevice, ctx->stream);
  };
  PGC_CK(ctx, copy_in(ctx->w, p));
  p += Kd;
  for (int64_t r = 0; r < (int64_t)ctx->owners * ctx->c; ++r, p += Kd) PGC_CK(ctx, copy_in(ctx->store + r * ctx->P, p));
  for (int o = 0; o < ctx->c; ++o, p += Kd) PGC_CK(ctx, copy_in(ctx->U + (int64_t)o * ctx->P, p));
  if (ctx->wb) PGC_CK(ctx, launch_f32_to_bf16(ctx->w, ctx->wb, ctx->P, ctx->stream));
  const int rc = read_status(ctx);
  if (rc) return rc;
  ctx->t = h[11];
  ctx->stepped = h[12] != 0;
  return PGC_OK;
}

int64_t pgc_step_count(const pgc_ctx* ctx) { return ctx ? ctx->t : -1; }

int pgc_timing(pgc_ctx* ctx, int32_t enable) {
  if (!ctx) return PGC_EINVAL;
  PGC_CK(ctx, cudaStreamSynchronize(ctx->stream));
  ctx->timing = enable != 0;
  if (enable) {
    ctx->ev_used = 0;
    ctx->timed_steps = 0;
    for (int k = 0; k < PGC_NKGROUPS; ++k) ctx->launches[k] = 0;
  }
  return PGC_OK;
}

int pgc_timing_read(pgc_ctx* ctx, double* ms, int64_t* launches, int64_t* steps_out) {
  if (!ctx) return PGC_EINVAL;
  PGC_CK(ctx, cudaStreamSynchronize(ctx->stream));
  double acc[PGC_NKGROUPS] = {0, 0, 0, 0, 0};
  // PGC_NKGROUPS + 1 events per recorded step: before the first group and after each
  for (size_t i = 0; i + PGC_NKGROUPS < ctx->ev_used; i += PGC_NKGROUPS + 1) {
    for (int k = 0; k < PGC_NKGROUPS; ++k) {
      float t = 0.f;
      PGC_CK(ctx, cudaEventElapsedTime(&t, ctx->ev_pool[i + k], ctx->ev_pool[i + k + 1]));
      acc[k] += t;
    }
  }
  if (ms)
    for (int k = 0; k < PGC_NKGROUPS; ++k) ms[k] = acc[k];
  if (launches)
    for (int k = 0; k < PGC_NKGROUPS; ++k) launches[k] = ctx->launches[k];
  if (steps_out) *steps_out = ctx->timed_steps;
  return read_status(ctx);
}

}  // extern "C"
