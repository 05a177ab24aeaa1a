/*
 * pgc.h — C ABI of libpgc, the GB300 (sm_103a) hot path of Pipelined
 * Gradient Coding (PGC).
 *
 * One GPU simulates an n-worker PGC training step that tolerates s
 * stragglers (c = s + 1 partitions per worker).  Every call is ordered on the
 * CUDA stream given to pgc_create.  A context is not thread-safe.
 *
 * Status codes: every int-returning call returns PGC_OK (0) or a negative
 * PGC_E* code; pgc_strerror turns a code into text.  On any error the
 * context's state (step counter, parameters, stores) is unchanged, except for
 * PGC_ECUDA / PGC_ETIMEOUT which leave the context unusable (destroy it).
 *
 * Layouts: features of partition D_k are row-major [m_k][d] (fp32 or bf16
 * bits); labels are float32 [m_k] (logistic: 0/1, least squares: real) or
 * int32 [m_k] class indices (softmax).  Parameters beta are float32 [K][d]
 * row-major (K = 1 for logistic and least squares).
 */
#ifndef PGC_H_
#define PGC_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define PGC_OK        0
#define PGC_EINVAL   (-1)  /* bad argument (sizes, enum, NULL pointer)       */
#define PGC_EMASK    (-2)  /* straggler mask is not exactly s ones, n-s zeros */
#define PGC_ESTATE   (-3)  /* call out of order (e.g. step before load)      */
#define PGC_ENOMEM   (-4)  /* device or pinned-host allocation failed        */
#define PGC_ECUDA    (-5)  /* a CUDA runtime call or kernel failed           */
#define PGC_ENOTSUP  (-6)  /* valid but unsupported combination             */
#define PGC_ETIMEOUT (-7)  /* a bounded device-side wait gave up            */
#define PGC_ESCRATCH (-8)  /* problem larger than pgc_gradient_noalloc's
                              fixed scratch                                 */
#define PGC_ESINGULAR (-9) /* GC-CR: the draws leave a worker's encoding
                              system singular, or the encoding cannot decode
                              the straggler set                             */

/* ---- enumerations (passed as int32) ------------------------------------ */
/* Dataset placement, §III: FR needs c | n; CR places cyclically.          */
#define PGC_FR 0
#define PGC_CR 1
/* Per-sample loss f: logistic cross-entropy (y in {0,1}), least squares
 * (1/2)(x.beta - y)^2, softmax cross-entropy over K classes.             */
#define PGC_LOGISTIC 0
#define PGC_LSQ      1
#define PGC_SOFTMAX  2
/* Storage type of the features.                                           */
#define PGC_F32  0
#define PGC_BF16 1

typedef struct pgc_ctx pgc_ctx;

/* Filled by pgc_step.  The arrays are owned by the caller and may be NULL. */
typedef struct pgc_step_info {
  int64_t  t;               /* index of the step just taken (0 = warm-up)    */
  int32_t  slot;            /* o_t = (t - 1) mod c written this step; -1 at t = 0 */
  int32_t  received;        /* n - s coded gradients decoded                 */
  int32_t *eval_partition;  /* [n]: partition W_i evaluated; -1 at t = 0     */
  int32_t *fr_rep;          /* [n/c] (FR only): worker that represents group j */
} pgc_step_info;

/*
 * pgc_create — allocate a PGC run (§III problem statement, §IV-A, §V-B).
 *   out      : receives the context (set to NULL on error).
 *   n, s     : workers and tolerated stragglers; 1 <= c = s + 1 <= n; FR
 *              additionally needs c | n.  n <= 1024.
 *   scheme   : PGC_FR or PGC_CR.   loss: PGC_LOGISTIC, PGC_LSQ, PGC_SOFTMAX.
 *   dtype    : storage of the features (PGC_F32 or PGC_BF16).
 *   d        : features per sample (>= 1).  K: classes (1 unless softmax;
 *              softmax needs 2 <= K <= 4096).
 *   rows     : host array [n], rows m_k >= 1 of partition D_k.
 *   lr       : learning rate eta of beta <- beta - eta * ghat (§III).
 *   w0       : host array [K*d] initial beta, or NULL for zeros.
 *   stream   : cudaStream_t every call is ordered on (NULL = legacy stream).
 * Allocates all device state (partitions, parameters, the per-owner gradient
 * stores, slot totals, scratch).  Errors: PGC_EINVAL, PGC_ENOTSUP,
 * PGC_ENOMEM, PGC_ECUDA.  Argument checks happen before any CUDA call.
 */
int pgc_create(pgc_ctx **out, int32_t n, int32_t s, int32_t scheme, int32_t loss,
               int32_t dtype, int64_t d, int64_t K, const int64_t *rows, float lr,
               const float *w0, void *stream);

/* Training schemes on the same kernels (§VI-A, the paper's baselines). */
#define PGC_MODE_PGC    0   /* pipelined gradient coding (default)                  */
#define PGC_MODE_IS_SGD 1   /* ignore stragglers: worker W_i evaluates D_i each step;
                               the master averages the n - s received gradients.
                               Needs scheme PGC_CR (the decode runs as CR with one
                               slot per worker, coefficient 1/(n - s)).             */
#define PGC_MODE_GC     2   /* gradient coding (GC, §VI-A): every worker evaluates
                               all c of its partitions each step.  PGC_FR: the
                               master decodes one coded gradient per group (1/n),
                               which recovers (1/n) sum_k g_k exactly.  PGC_CR:
                               GC-CR (§V-A), worker W_j uploads
                               sum_l c_{j,l} g_{(j+l) mod n} with the encoding of
                               pgc_set_gc_encoding and the master applies the
                               decode weights d_m(J) of the received set, times
                               1/n: exact as well.  PGC_CR needs n <= 64.        */
#define PGC_MODE_NAIVE_CR 3 /* the naive pipelined construction on cyclic
                               repetition (§V-A): PGC-CR's rotation and stores
                               (one partition evaluated per step), but W_j uploads
                               sum_l c_{j,l} (its latest gradient of
                               D_{(j+l) mod n}) and the master decodes with GC-CR's
                               weights d_m(J), times 1/n.  Stale copies enter with
                               the decoding coefficients alpha_{m,k} = d_m c_{j_m,l}
                               (pgc_get_gc_decode).  Needs PGC_CR and n <= 64.   */

/*
 * pgc_create_mode — pgc_create with a training scheme from PGC_MODE_*; the
 * other arguments and errors are pgc_create's (PGC_EINVAL also for an unknown
 * mode or a mode/scheme pair listed as unsupported above).  With s = 0 every
 * mode is plain distributed gradient descent (DGD, §III).
 */
int pgc_create_mode(pgc_ctx **out, int32_t mode, int32_t n, int32_t s, int32_t scheme, int32_t loss,
                    int32_t dtype, int64_t d, int64_t K, const int64_t *rows, float lr,
                    const float *w0, void *stream);

/*
 * pgc_set_gc_encoding — GC-CR's encoding coefficients c_{j,l} (§V-A), for the
 * modes that decode with them (PGC_MODE_NAIVE_CR; PGC_MODE_GC with PGC_CR).
 * §V-A takes them from gradient coding's cyclic-repetition construction,
 * which the device builds from the given random numbers: H = [draws |
 * -(row sums of draws)] is s x n with H 1 = 0; worker W_j's row of the
 * encoding matrix B is supported on partitions j..j+s (mod n), has
 * c_{j,0} = B[j][j] = 1, and its other s entries solve
 * H[:, {j+1..j+s}] x = -H[:, j] (fp64, partial pivoting).
 *   draws : host array [s][n-1], row-major (for instance standard normal
 *           draws); ignored when s = 0 (then B is the identity).
 * Must be called before the first pgc_step of those modes (PGC_ESTATE
 * otherwise); may be called again.  Not part of a checkpoint.  Errors:
 * PGC_EINVAL (other mode, NULL or non-finite draws), PGC_ESINGULAR (a
 * worker's system is singular; the context stays usable), PGC_ECUDA.
 */
int pgc_set_gc_encoding(pgc_ctx *ctx, const double *draws);

/*
 * pgc_get_gc_encoding — copy the encoding coefficients to host coeff[n][c]:
 * coeff[j*c + l] = c_{j,l}, W_j's weight on its gradient of D_{(j+l) mod n}.
 * Errors: PGC_EINVAL (other mode), PGC_ESTATE (not set), PGC_ECUDA.
 */
int pgc_get_gc_encoding(pgc_ctx *ctx, double *coeff);

/*
 * pgc_get_gc_decode — what the device derived at the last step of a GC-CR
 * mode (§V-A): d (host [n], or NULL) = the decode weights d_j(J) solving
 * sum_{j in J} d_j B[j] = 1 over the received set J (0 for stragglers), in
 * fp64; alpha_range (host [2], or NULL) = the maximum and the minimum of the
 * decoding coefficients alpha_{m,k} = d_m c_{j_m,l} over the received workers
 * and the partitions each holds.  The decoded gradient is
 * (1/n) sum_j d_j sum_l c_{j,l} store[j][l].  A straggler set the encoding
 * cannot decode (sum_j d_j B[j] misses 1 by more than 1e-8 relative, or a
 * pivot vanishes) leaves that step's beta unchanged and makes the call that
 * reads the device status (pgc_step with host outputs, pgc_sync) return
 * PGC_ESINGULAR; the context then takes no more steps.  Errors: PGC_EINVAL,
 * PGC_ESTATE (no step yet), PGC_ECUDA.
 */
int pgc_get_gc_decode(pgc_ctx *ctx, double *d, double *alpha_range);

/*
 * pgc_load_partitions — copy the n partitions into device memory (§III: the
 * partitions are placed before training).  X[k] points to [m_k][d] features
 * of the create-time dtype, y[k] to m_k labels (float32, or int32 for
 * softmax).  on_device != 0: the pointers are device pointers; otherwise host
 * pointers.  The library keeps its own copy; the caller may free its buffers
 * after the call returns.  May be called again to replace the data; it does
 * not reset the step counter.  Errors: PGC_EINVAL (NULL entry), PGC_ECUDA.
 */
int pgc_load_partitions(pgc_ctx *ctx, const void *const *X, const void *const *y,
                        int32_t on_device);

/*
 * pgc_step — one PGC training step t (§IV-A PGC-FR, §V-B PGC-CR).
 *   straggler_mask : host array [n]; 1 marks a straggler, 0 a worker whose
 *                    coded gradient reaches the master.  Exactly s ones.
 *   grad_out       : [K*d] float32, receives the decoded gradient ghat^(t)
 *                    (NULL: not returned).
 *   w_out          : [K*d] float32, receives beta^(t+1) (NULL: not returned).
 *   outputs_on_device : != 0: grad_out / w_out are device pointers and the
 *                    call returns without waiting for the GPU; 0: host
 *                    pointers, the call waits until they hold the results
 *                    (pinned host buffers mapped into the device's address
 *                    space and 16-byte aligned are written by the decode
 *                    kernel itself when the parameter rows need no padding;
 *                    others are filled by copies after it).
 *   info           : may be NULL; receives t, o_t and the schedule indices.
 * Step 0 is the warm-up: every worker evaluates all c of its partitions at
 * beta^(0).  From step 1 on, worker W_i evaluates only the partition in its
 * slot o_t = (t-1) mod c; stragglers still evaluate and store.  FR workers of
 * one group evaluate the same partition at the same beta, so it is computed
 * once per group.  The decode uses the coded gradients of the n - s received
 * workers with the coefficients of §IV-A (FR: one per group, times 1/n) or
 * §V-B (CR: times 1/((n-s)c)), derived on the device from the mask, and is
 * fused with the SGD update.  Errors: PGC_ESTATE (no partitions loaded),
 * PGC_EMASK, PGC_EINVAL, PGC_ECUDA, PGC_ETIMEOUT.
 */
int pgc_step(pgc_ctx *ctx, const uint8_t *straggler_mask, float *grad_out, float *w_out,
             int32_t outputs_on_device, pgc_step_info *info);

/*
 * pgc_loss — F(beta^(t)) = (1 / sum_k m_k) sum over all samples of f, at the
 * current parameters (§III).  Untimed helper; waits for the GPU.
 * Errors: PGC_ESTATE, PGC_EINVAL, PGC_ECUDA.
 */
int pgc_loss(pgc_ctx *ctx, double *loss_out);

/*
 * pgc_sync — wait for every call issued on the context's stream and report
 * a device-side failure (PGC_ETIMEOUT if a bounded wait gave up, PGC_EMASK
 * if the decode kernel saw an invalid mask).  Steps with device outputs do
 * not wait; call this before trusting their results.
 */
int pgc_sync(pgc_ctx *ctx);

/* pgc_destroy — free everything; NULL is accepted.  Returns PGC_OK. */
int pgc_destroy(pgc_ctx *ctx);

/* pgc_strerror — static text for a status code. */
const char *pgc_strerror(int32_t code);

/* pgc_gradient_path — static name of the kernel path the context computes
 * per-partition gradients with (fixed at pgc_create): "grad_rows" (logistic,
 * least squares), "tc_fused" (softmax on the tensor cores, residual in the
 * logits GEMM), "tc" (tensor cores, separate residual kernel),
 * "softmax_rows" (few classes, whole rows per CTA pair), "softmax_cluster" (few
 * classes, 8-CTA clusters), "softmax_cc" (CUDA cores); "" for NULL. */
const char *pgc_gradient_path(const pgc_ctx *ctx);

/* pgc_last_cuda_error — name of the CUDA runtime error behind the most
 * recent PGC_ECUDA / PGC_ENOMEM returned on the calling thread (for example
 * "cudaErrorLaunchOutOfResources"), or "" if there was none.  Static text. */
const char *pgc_last_cuda_error(void);

/* ---- host-only helpers: pure index arithmetic, no CUDA call ------------- */

/*
 * pgc_placement — the partitions each worker holds (§III; §IV-A for FR,
 * §V-B for CR), table[i*c + l] = partition in slot l of worker W_i.
 * table: host [n*c].  Errors: PGC_EINVAL.
 */
int pgc_placement(int32_t scheme, int32_t n, int32_t s, int32_t *table);

/*
 * pgc_schedule — partition each worker evaluates at step t (§IV-A, §V-B):
 * eval_partition[i] (host [n]) = the partition in slot (t-1) mod c of W_i,
 * or -1 for every worker at t = 0; *slot = (t-1) mod c or -1.
 * Errors: PGC_EINVAL.
 */
int pgc_schedule(int32_t scheme, int32_t n, int32_t s, int64_t t,
                 int32_t *eval_partition, int32_t *slot);

/* ---- inspection of device state (tests; each call waits for the GPU) ---- */

/*
 * pgc_get_store — copy worker W_i's stored gradient in slot l (the gradient
 * of the partition in slot l of its holdings, as last evaluated) to host
 * out[K*d].  FR workers of one group share one store.  Errors: PGC_EINVAL,
 * PGC_ESTATE, PGC_ECUDA.
 */
int pgc_get_store(pgc_ctx *ctx, int32_t worker, int32_t slot, float *out);

/*
 * pgc_get_store_cols — as pgc_get_store, for the parameters [col0, col0 +
 * ncols) of the flattened K*d vector only (host out[ncols]); reads a few
 * columns of every store without copying whole gradients.  Errors:
 * PGC_EINVAL (range outside [0, K*d)), PGC_ESTATE, PGC_ECUDA.
 */
int pgc_get_store_cols(pgc_ctx *ctx, int32_t worker, int32_t slot, int64_t col0, int64_t ncols, float *out);

/*
 * pgc_get_decode — the decoding coefficients the device derived from the
 * last step's mask: coeff[i] (host [n]) = weight a_i of W_i's coded gradient
 * (§IV-A: 1/n for each FR group's representative; §V-B: 1/((n-s)c) for each
 * received CR worker; GC-CR modes: d_i(J)/n; 0 otherwise).  Errors:
 * PGC_ESTATE, PGC_ECUDA.
 */
int pgc_get_decode(pgc_ctx *ctx, float *coeff);

/* pgc_get_weights — copy the current beta to host out[K*d]. */
int pgc_get_weights(pgc_ctx *ctx, float *out);

/* pgc_set_weights — overwrite beta with host w[K*d] (teacher forcing in
 * tests; also the checkpoint-restore path).  Errors: PGC_EINVAL, PGC_ECUDA. */
int pgc_set_weights(pgc_ctx *ctx, const float *w);

/*
 * Checkpoint and resume of a run: the step counter t, beta, every store
 * (owners x c gradients) and the slot totals U — everything a later step
 * reads.  The features and labels are not part of it: the resumed context
 * must be created with the same arguments and loaded with the same
 * partitions.
 *
 * pgc_checkpoint_bytes — *bytes = size of the checkpoint of this context:
 *   104 bytes of header (13 int64: magic 0x3154504B43434750 "PGCCKPT1",
 *   version 1, mode, scheme, loss, dtype, n, s, c, d, K, t, stepped) then fp32
 *   beta [K][d], stores [owners][c][K][d] and U [c][K][d], host byte order.
 * pgc_checkpoint_save — write it to host buf[bytes] (waits for the stream).
 * pgc_checkpoint_load — restore it from host buf[bytes] into a context with
 *   the same mode, scheme, loss, dtype, n, s, d and K; the next pgc_step is
 *   step t of the saved run.
 * Errors: PGC_EINVAL (NULL, wrong size, header of another configuration),
 * PGC_ESTATE (a failed context), PGC_ECUDA.
 */
int pgc_checkpoint_bytes(pgc_ctx *ctx, int64_t *bytes);
int pgc_checkpoint_save(pgc_ctx *ctx, void *buf, int64_t bytes);
int pgc_checkpoint_load(pgc_ctx *ctx, const void *buf, int64_t bytes);

/* pgc_step_count — number of steps taken so far (host-side counter). */
int64_t pgc_step_count(const pgc_ctx *ctx);

/* ---- measurement ---------------------------------------------------------- */

/* Kernel groups of one step, in launch order, as counted and timed below.
 * Paths without a group leave it empty (zero time, zero launches). */
#define PGC_KGRAD   0   /* gradient: streaming row kernel, few-class softmax
                           kernel, tensor-core logits GEMM, or the CUDA-core
                           softmax kernels                                     */
#define PGC_KRESID  1   /* tensor-core softmax: residual R = softmax(Z) - Y    */
#define PGC_KGRADB  2   /* tensor-core softmax: gradient GEMM R^T X            */
#define PGC_KCOMMIT 3   /* gradient-store commit                               */
#define PGC_KDECODE 4   /* decode coefficients + decode + SGD                  */
#define PGC_NKGROUPS 5

/*
 * pgc_timing — enable != 0 starts recording CUDA events on the context's
 * stream around each kernel group of every following step (and clears what
 * was recorded); 0 stops.  Errors: PGC_EINVAL, PGC_ECUDA.
 */
int pgc_timing(pgc_ctx *ctx, int32_t enable);

/*
 * pgc_timing_read — wait for the stream, then return for each kernel group
 * the summed device time in milliseconds (ms[PGC_NKGROUPS]) over the steps
 * recorded since timing was enabled, and the kernels launched by the library
 * in those steps (launches[PGC_NKGROUPS]).  Either array may be NULL.
 * *steps_out (nullable) receives the number of recorded steps.
 */
int pgc_timing_read(pgc_ctx *ctx, double *ms, int64_t *launches, int64_t *steps_out);

/* ---- allocation-free gradient --------------------------------------------- */

/*
 * pgc_gradient_noalloc — g_out = (1/m) sum over the m rows x of one partition
 * of r(x) * x, with r = sigmoid(x.w) - y (PGC_LOGISTIC) or x.w - y (PGC_LSQ):
 * the per-partition gradient pgc_step evaluates, computed without allocating
 * any device memory.  The paper has no counterpart; this exists for callers
 * that cannot call cudaMalloc / cudaFree when they need a gradient: a
 * framework whose caching pool already holds the free device memory, or a
 * loop that must not take cudaFree's implicit device synchronisation.
 *
 *   X     : device [m][d] features (PGC_F32, or PGC_BF16 bits), 16-byte aligned
 *   y     : device [m] float32 labels;  w: device [d] float32 parameters
 *   g_out : device [d] float32, 16-byte aligned (written)
 *   stream: cudaStream_t to run on; the call waits for it before returning.
 *
 * Scratch: a fixed 16 MiB array inside the library (a __device__ global),
 * held on every GPU that loads the library until the process exits.  The
 * first call on a device looks up the array's device address (with that
 * device current) and keeps it for the life of the process; make that first
 * call before any stream capture.  cudaDeviceReset on a device unloads the
 * library's module there and makes the kept address stale: a process that
 * resets a device must not call this entry point on it afterwards.  All
 * calls share the array and it keeps the last call's contents; each call
 * rewrites what it reads, but calls that overlap on the GPU (other streams,
 * other threads) race on it.
 *
 * Limits: d must be a row length the gradient kernel takes without padding
 * (fp32: 32, 64, 128 * 2^k up to 16384; bf16: 64, 128, 256 * 2^k up to
 * 32768), else PGC_ENOTSUP.  The scratch holds a copy of the m labels (4 m
 * bytes) and one partial sum of 4 d bytes per SM; problems that do not fit
 * the 16 MiB return PGC_ESCRATCH (on a 152-SM GPU: about 1.7 million rows at
 * fp32 d = 16384, about 4 million at d = 1024).  Other errors: PGC_EINVAL,
 * PGC_ECUDA, PGC_ETIMEOUT.
 */
int pgc_gradient_noalloc(int32_t loss, int32_t dtype, int64_t m, int64_t d, const void *X,
                         const float *y, const float *w, float *g_out, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* PGC_H_ */
