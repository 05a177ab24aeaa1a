// Internal interfaces between the host control code (pgc_api.cu) and the
// kernel files.  Nothing here is part of the public ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace pgc {

// Error bits written to a context's device status word.
enum : int {
  kErrWaitTimeout = 1,   // a bounded mbarrier wait gave up
  kErrBadMask = 2,       // the decode kernel saw a mask with popcount != s
  kErrBadShape = 4,      // a kernel was launched with an impossible shape
  kErrSingular = 8,      // GC-CR: the draws cannot encode, or the straggler set cannot be decoded
};

// A contiguous row range of one evaluated partition, processed by one CTA.
// Rows are global row indices into the packed feature buffer (all partitions
// back to back, each row padded to `ld` elements).
struct WorkItem {
  int32_t e;        // position of the partition in the phase's evaluated list
  int32_t part;     // partition index k
  int64_t row0;     // first global row
  int64_t rows;     // number of rows (>= 1)
};

// ---- K5 + K6: decode coefficients from the mask, decode, SGD --------------
constexpr int kMaxWorkers = 1024;
// softmax on the tensor cores from this many classes on (the forward N tile is
// 256 classes; below half a tile the padding outweighs the tensor-core gain)
constexpr int64_t kTcMinClasses = 128;
constexpr int64_t kTcMaxClasses = 2048;   // the residual kernel keeps a row in registers
struct MaskBits {
  uint32_t w[kMaxWorkers / 32];
};
struct DecodeArgs {
  int scheme, n, s, c;
  int slot;                 // o_t refreshed this step, or -1: all slots (warm-up)
  int owners;               // stores: n (CR) or n / c (FR groups)
  MaskBits mask;            // bit i = 1: worker i straggles
  int64_t P;                // floats per gradient (multiple of 4)
  float* store;             // [owners * c][P]
  float* U;                 // [c][P] slot totals
  float* w;                 // [P] parameters, updated in place
  uint16_t* wb;             // [P] bf16 copy of w, or nullptr
  float* gout;              // [P] decoded gradient
  float lr;
  float* coeff_out;         // [n] per-worker coefficient a_i (written once per step)
  int* status;
  float* g_user = nullptr;  // optional extra destinations of ghat and beta, same
  float* w_user = nullptr;  // unpadded layout (used when ld == d)
  int u_ready = 0;          // U[slot] already holds this step's slot total
  const float* pre = nullptr;  // with u_ready: the terms of the slots other than o_t, summed
                               // early (TcSoftmaxParams::pre_out)
};
// ---- K1: streaming gradient of logistic / least-squares partitions -------
// For every work item: partial[item][0:ld] = sum over its rows x of
// residual(x) * x, residual = sigmoid(x.w) - y (logistic) or x.w - y (lsq).
struct GradRowsArgs {
  int loss;                 // PGC_LOGISTIC or PGC_LSQ
  int dtype;                // PGC_F32 or PGC_BF16
  int64_t d, ld;            // features, padded row length (elements)
  const void* X;            // packed features [total_rows][ld]
  const float* y;           // packed labels [total_rows]
  const float* w;           // parameters [ld] (padding is zero)
  const WorkItem* items;    // device [nitems]
  int nitems;
  int max_item_rows;        // rows of the largest item
  float* partials;          // [nitems][ld]
  // Labels are copied per stage from a 16-byte aligned start, so up to 12
  // bytes past the last label are read: y must be padded by 16 bytes.
  // Dynamic scheduling: with work_ctr set, `grid` persistent CTAs take items
  // blockIdx.x, then gridDim.x + atomicAdd(work_ctr, 1); the last producer
  // resets work_ctr and prod_done.  Without it, one CTA per item.
  int* work_ctr = nullptr;
  int* prod_done = nullptr;
  int grid = 0;
  int* status;              // device status word (error bits)
  // Fused tail.  tail = 0: partial sums only.  1: the last CTA of each
  // partition also commits it (ordered sum of its partials, scaled, into its
  // destination stores).  2: additionally the CTA committing the last
  // partition derives the decode coefficients, decodes and updates w (dec).
  int tail = 0;
  bool pdl = false;         // programmatic dependent: consumers wait before reading w
  int* cnt_e = nullptr;     // [nE] arrivals per partition, zero between steps
  int* cnt_all = nullptr;   // committed partitions, zero between steps
  const int32_t* e_item0 = nullptr;
  const float* e_scale = nullptr;
  const int32_t* e_dest = nullptr;
  int ndest = 1;
  int nE = 0;
  float* store = nullptr;   // [owners * c][ld]
  DecodeArgs dec;           // used when tail == 2
  int64_t prefetch_bytes = 0; // L2 warm-up per CTA before waiting for the previous step
};
int grad_rows_variant(int dtype, int64_t d, int64_t* ld_out);  // chooses ld, returns variant id
int grad_rows_stage_rows(int variant, int64_t ld, int dtype);
cudaError_t launch_grad_rows(const GradRowsArgs& a, int variant, cudaStream_t st);

// ---- K4: partial reduction + store commit ----------------------------------
// For each evaluated partition e (CSR over items): g = scale[e] * sum of its
// items' partials (in item order), written to every destination store
// dest[e*ndest + j] (an index owner*c + slot, or -1 for none).
struct CommitArgs {
  const float* partials;    // [nitems][P]
  int64_t P;                // floats per gradient (K * ld), multiple of 4
  const int32_t* e_item0;   // [nE + 1]
  const float* e_scale;     // [nE] 1 / m_e
  const int32_t* e_dest;    // [nE * ndest]
  int ndest;
  int nE;
  float* store;             // [owners * c][P]
};
cudaError_t launch_commit(const CommitArgs& a, cudaStream_t st, bool pdl = false);

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st, bool pdl, int sm_count);

// ---- GC-CR coding: the naive pipelined construction and GC-CR (§V-A) -------
constexpr int kGcMaxN = 64;   // workers of the GC-CR modes (one-warp fp64 solves)
struct GcWeightsArgs {
  int n, s, c;
  MaskBits mask;
  const double* coeff;      // [n][c] encoding coefficients c_{j,l}
  double* d;                // [n] decode weights d_j(J), 0 for stragglers
  float* wts;               // [n][c] d_j c_{j,l} / n, applied to store[j][l]
  float* coeff_out;         // [n] d_j / n, the weight of W_j's coded gradient
  double* alpha;            // [2] max and min of alpha_{m,k} = d_m c_{j_m,l}
  int* status;
};
// Encoding coefficients [n][c] from draws [s][n-1] (device); one launch.
cudaError_t launch_gc_encoding(const double* draws, int n, int s, double* coeff, int* status, cudaStream_t st);
// The step's decode weights (one CTA), then decode + SGD over the stores
// (programmatic dependent of the weights kernel when pdl is set).
cudaError_t launch_gc_decode(const GcWeightsArgs& w, const DecodeArgs& a, cudaStream_t st, bool pdl, int sm_count);

// ---- generic softmax gradient on CUDA cores --------------------------------
// logits Z[r][k] = sum_j W[k][j] x_r[j] for the rows of each evaluated
// partition, then R = softmax(Z) - onehot(y) in place, then
// partial[e][k*ld + j] = sum_{r in e} R[r][k] x_r[j].
struct SoftmaxCCArgs {
  int dtype;
  int64_t ld, K;
  const void* X;            // packed [total_rows][ld]
  const int32_t* y;         // packed class labels
  const float* W;           // [K][ld]
  const int64_t* e_row0;    // [nE] global first row of each evaluated partition
  const int64_t* e_rows;    // [nE]
  const int64_t* e_zrow0;   // [nE] first row of the partition in Z
  int nE;
  int64_t max_rows;         // max rows of an evaluated partition
  int64_t z_total;          // rows of Z (sum of the evaluated partitions' rows)
  float* Z;                 // scratch [z_total][Kpad]
  int64_t Kpad;
  float* partials;          // [nE][K*ld]
};
cudaError_t launch_softmax_cc(const SoftmaxCCArgs& a, cudaStream_t st);

// ---- full loss ------------------------------------------------------------
// Per-row f summed in fp64 into blocksum[block]; a second pass adds them in
// block order.
struct LossArgs {
  int loss, dtype;
  int64_t ld, K, rows;      // all rows of all partitions
  const void* X;
  const void* y;            // float (logistic/lsq) or int32 (softmax)
  const float* w;           // [K][ld]
  double* blocksum;         // scratch [nblocks]
  int nblocks;
  double* out;              // device double
  // softmax only: logits are formed in row chunks
  float* Z;                 // scratch [z_chunk_rows][Kpad]
  int64_t Kpad;
  int64_t z_chunk_rows;
  const int64_t* chunk_desc; // device [3 * nchunks]: {row0, rows, 0} per chunk
};
cudaError_t launch_loss(const LossArgs& a, cudaStream_t st);

// ---- tensor-core logits GEMM (tc_gemm.cu) --------------------------------
// Z[r][k] = sum_j X[r][j] Wb[k][j] (A = X K-major, B = Wb K-major), for the
// class counts the fused logits + residual kernel does not cover.
struct TcGemmParams {
  int nbatch;
  const int* tile_prefix;   // [nbatch + 1] pair tiles before batch b (ceil(MT_b / 2) * NT each)
  const int* mt_count;      // [nbatch] row tiles (of 128) MT_b
  int NT;                   // class tiles (of 256) per batch
  const int* nk;            // [nbatch] K blocks (of 64)
  const int* a_off;         // [nbatch] first X row of the batch
  int total_tiles;
  // Results leave through TMA stores of 32 x 32 fp32 boxes into the 2-D map
  // Z [rows][Kpad], box at (n, out_row0[b] + m).
  const int64_t* out_row0;  // first Z row of batch b (a multiple of 128)
  int* status;
  int pdl;
};
// Tensor maps (tm_out: 128 bytes, 64-byte aligned, a CUtensorMap), 128-byte
// swizzle, out-of-range elements read as zero and are not written.
// bf16 2-D [outer][inner], box {64, box_outer}
bool make_tmap_bf16(void* tm_out, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
                    uint32_t box_outer);
// fp32 rank-2 or rank-3 (dims innermost first, byte strides of dims 1..), box {32, 32, 1}
bool make_tmap_f32_box32(void* tm_out, const void* base, int rank, const uint64_t* dims, const uint64_t* strides);
cudaError_t launch_tc_gemm(const void* tmA, const void* tmB, const void* tmOut, const TcGemmParams& p, int grid,
                           cudaStream_t st);
// R = softmax(Z) - onehot(y) as bf16, zero for classes K..Kpad-1 and for the
// rows up to the next multiple of 64; also zeroes zero_buf[0:zero_n] (floats,
// a multiple of 4) when given.
cudaError_t launch_softmax_bf16(const float* Z, uint16_t* Rb, int64_t Kpad, int64_t K, const int32_t* y,
                                const int64_t* e_row0, const int64_t* e_rows, const int64_t* e_zrow0, int nE,
                                int64_t max_rows, float* zero_buf, int64_t zero_n, cudaStream_t st);

// ---- tensor-core gradient contraction (tc_grad.cu) -------------------------
// G_e = scale_e R_e^T X_e for the runs of partitions in `units`
// ({class pair tile mp, feature tile nt, first batch, batches}), written into
// the stores [slot][K][ld] at every dest of the batch (TMA tensor stores
// through tmS); with u_reduce each
// run's sum is also added (TMA reduce-add, fp32 box 32 x 32 x 1) into
// U [c][K][ld] at u_slot.  R is read as MN-major A (box 64 x 64), X as
// MN-major B (box 64 x 64).
struct TcGradParams {
  const int4* units;
  int nunits;
  const int* nk;            // [nbatch] K blocks of 64 rows (ceil(m_e / 64))
  const int* a_off;         // [nbatch] first R row of the batch
  const int* b_off;         // [nbatch] first X row of the batch
  const float* scale;       // [nbatch] 1/m_e
  const int32_t* dest;      // [nbatch * ndest] store index or -1
  int ndest;                // destinations: the stores, through the tmS tensor map
  int m_limit;              // classes that exist (K); rows past it are not written
  int u_reduce;
  int u_slot;
  int* status;
  int pdl;
};
constexpr int kTcGradMaxRun = 8;   // partitions per unit at most
// Clusters of two that fit at once (0: the kernel cannot be launched).
int tc_grad_max_pairs();
// tmS: the stores [owners * c][K][ld] fp32, box 32 x 32 x 1 (written by TMA)
cudaError_t launch_tc_grad(const void* tmR, const void* tmX, const void* tmU, const void* tmS, const TcGradParams& p,
                           int npairs, cudaStream_t st);

// ---- tensor-core logits GEMM with the softmax residual in its epilogue ------
// (tc_softmax.cu) for every 128-row tile {first X row, first R row, valid
// rows, partition}: R[r][k] = softmax_k(X Wb^T)[r] - [k == y_r] as bf16, rows
// past `valid` zero.  A cluster of NT = Ktc / 256 CTAs (1, 2, 4 or 8) covers
// all classes of one tile; also zeroes zero_buf[0 : 4 zero_n4].
struct TcSoftmaxParams {
  const int4* tiles;
  int ntiles;
  int NT;                   // CTAs per cluster (256 classes each)
  int nk;                   // ld / 64
  int K;
  const int32_t* y;         // labels per global X row
  float* zero_buf;
  int64_t zero_n4;
  int* status;
  int pdl;
  // Early part of the step's decode (steady steps, U[o_t] formed by the
  // gradient contraction): with pre_out set, the grid also writes
  // pre_out[p] = B sum_{o != o_t} U[o][p] + sum_{deviating stores r}
  // (b_r - B) sum_{o != o_t} store[r][o][p] for every float4 column p
  // (pre: the step's decode arguments); the decode then adds the slot o_t
  // terms (DecodeArgs::pre).
  DecodeArgs pre;
  float* pre_out = nullptr;
};
// Columns (float4) from which the step's decode is split this way, and the
// deviating stores (CR: stragglers) it handles at most.
constexpr int64_t kPreDecodeMinP4 = 1 << 18;
constexpr int kPreMaxDev = 64;
// Clusters of NT that fit at once (0: this NT is not supported).
int tc_softmax_max_clusters(int NT);
// tmXq: X, box {64, 128 / NT}; tmW: Wb, box {64, 128}; tmR: Rb, box {64, 32}
cudaError_t launch_tc_softmax(const void* tmXq, const void* tmW, const void* tmR, const TcSoftmaxParams& p,
                              int nclusters, cudaStream_t st);

// ---- softmax with few classes: one pass over X per step --------------------
// tiles[i] = {first global X row, rows (<= kSmallKRows), item, flags: 1 first / 2 last
// tile of a cluster's run in one partition}; cluster c of nc takes tiles
// [ntiles c / nc, ntiles (c + 1) / nc).  partials[item][K][ld] receives the
// unscaled gradient sums of the run.
constexpr int kSmallKRows = 128;    // rows per tile of the few-class kernel
struct SmallKArgs {
  const int4* tiles;
  int ntiles;
  int nkb;                  // ld / 64
  int nper;                 // 64-feature blocks per CTA slice (ceil(nkb / 8))
  int K;
  const int32_t* y;         // labels per global row
  float* partials;
  int64_t P;                // K * ld
  int64_t ld;
  int* status;
  int pdl;
};
bool smallk_fits(int64_t K, int64_t ld);
int smallk_max_clusters(int nper);
cudaError_t launch_softmax_smallk(const void* tmX, const void* tmW, const SmallKArgs& a, int nclusters,
                                  cudaStream_t st);

// ---- softmax with few classes, whole rows per CTA pair (softmax_rows.cu) ---
// tiles[i] = {first global X row, rows (<= kRowsTileRows), item, flags: 1 first / 2 last
// tile of a pair's run in one partition}; pair p (a cluster of two CTAs, one
// per half of the features) takes tiles [pair_t0[p], pair_t0[p + 1]), a split
// made on the host that charges kRowsDrainTiles for each run starting inside
// a pair's range.
// partials[item][K][ld] receives the unscaled gradient sums of the run.
constexpr int kRowsTileRows = 16;
// A run (one partition's tiles) that starts inside a CTA pair's range stalls
// the pair's logits warps while the previous run drains: about this many
// tiles' time, charged when the host splits the tiles over the pairs.
constexpr int kRowsDrainTiles = 4;
constexpr int64_t kRowsMaxLd = 3072;       // the forward keeps a warp's W^T slice in registers
constexpr int kRowsMaxSlots = 8;
constexpr uint32_t kRowsSmemBudget = 227 * 1024 - 1024;   // a little static shared memory beside it
struct RowsArgs {
  const int32_t* pair_t0;   // [pairs + 1]: CTA pair p takes tiles [pair_t0[p], pair_t0[p + 1])
  const int4* tiles;
  int ntiles;
  int K;
  const int32_t* y;         // labels per global row
  const uint16_t* wb;       // bf16 W [16][ld], zero rows past K
  float* partials;
  int64_t P;                // K * ld
  int64_t ld;               // a multiple of 256, at most kRowsMaxLd
  int nslots;
  int box_blocks;           // 64-feature blocks per TMA copy (divides ld / 64)
  int* status;
  int pdl;
  // Fused tail (tail = 1): after a grid barrier every CTA commits, for its
  // slice of the float4 columns, every evaluated partition (ordered sum of the
  // partition's items, times e_scale, into each destination store), then
  // after a CTA barrier decodes and updates w (dec) over the same columns.
  // The grid must be co-resident (one CTA per SM); counters[0] and
  // counters[2] are zero between steps (the last CTA resets them).
  int tail = 0;
  int nE = 0;
  const int32_t* e_item0 = nullptr;  // [nE + 1]
  const float* e_scale = nullptr;    // [nE]
  const int32_t* e_dest = nullptr;   // [nE * ndest]
  int ndest = 1;
  float* store = nullptr;
  int* counters = nullptr;
  DecodeArgs dec;
};
// Slots of kRowsTileRows x ld/2 (a CTA's half tile) that fit (0: ld not supported).
int rows_slots(int64_t ld);
// 64-feature blocks per TMA copy: `requested` if it divides a half tile's
// blocks, else the largest such count up to 8.
int rows_box_blocks(int64_t ld, int requested);
// CTAs of the grid: two per co-resident cluster, one per SM (0: cannot launch).
int rows_max_ctas(int64_t ld, int nslots);
// tmX: X as [ld/64][rows][64] bf16 blocks, box {64, kRowsTileRows, box_blocks} (make_tmap_bf16_rows)
cudaError_t launch_softmax_rows(const void* tmX, const RowsArgs& a, int nctas, cudaStream_t st);
// 3-D view of a row-major bf16 [rows][ld] matrix as 64-element blocks: dims
// {64, rows, ld/64}, box {64, box_rows, box_blocks}, 128-byte swizzle; with
// tm_out and base both nullptr it only checks that the view can be encoded.
bool make_tmap_bf16_rows(void* tm_out, const void* base, uint64_t ld, uint64_t rows, uint32_t box_rows,
                         uint32_t box_blocks);

// ---- misc -------------------------------------------------------------------
cudaError_t launch_f32_to_bf16(const float* src, uint16_t* dst, int64_t count, cudaStream_t st);

}  // namespace pgc
