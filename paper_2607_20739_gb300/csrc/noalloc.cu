// pgc_gradient_noalloc: the gradient of one logistic or least-squares
// partition, computed with no device allocation at all.
//
// Who needs it: code that cannot call cudaMalloc / cudaFree at the point
// where it wants a gradient, for example a framework whose caching pool has
// already reserved the free device memory (so cudaMalloc would fail), or a
// latency-sensitive loop that must not pay for cudaFree's implicit device
// synchronisation.  The pgc_create path allocates its scratch once per
// context; this entry point instead uses one fixed scratch array that is
// part of the library image.
//
// How: the scratch lives in a file-scope __device__ array of
// kScratchBytes.  Every GPU that loads the library holds it until the process
// exits.  Host code cannot use the array's name as a device address, so the
// first call on each device, with that device current, looks the address up
// with cudaGetSymbolAddress and caches it; that first call should therefore
// come before any stream capture.  The cached address is not refreshed: after
// cudaDeviceReset (which unloads this module on that device) it is stale, so
// a process that resets a device must not call this entry point there again.  The call then fills its small work tables
// in the scratch with a kernel, runs the streaming gradient kernel (partial
// sums per CTA into the scratch) and the commit kernel (ordered sum of those
// partials, scaled by 1/m, into the caller's output), waits for the stream
// and reports a device-side failure.
//
// Sharing: every call uses the same array, which keeps what the last call
// left there.  Nothing in it has to start at zero (each call rewrites its
// tables and every partial it reads, and clears the status word it checks),
// but two calls whose work overlaps on the GPU, on different streams or host
// threads, race on the array and corrupt each other's results.
#include <algorithm>
#include <cstring>
#include <mutex>

#include "pgc.h"
#include "pgc_internal.h"

namespace {

constexpr size_t kScratchBytes = size_t(16) << 20;   // 16 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Scratch layout (bytes): [0,4) status word; [16,24) e_item0[2];
// [32,36) e_scale[1]; [48,52) e_dest[1]; [256, 256 + items) work items;
// then the per-CTA partial sums, 256-byte aligned.
constexpr size_t kOffStatus = 0, kOffItem0 = 16, kOffScale = 32, kOffDest = 48, kOffItems = 256;

size_t align256(size_t v) { return (v + 255) / 256 * 256; }

__global__ void noalloc_fill_tables(unsigned char* scratch, int G, int64_t m) {
  pgc::WorkItem* items = reinterpret_cast<pgc::WorkItem*>(scratch + kOffItems);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < G; i += gridDim.x * blockDim.x) {
    pgc::WorkItem it;
    it.e = 0;
    it.part = 0;
    it.row0 = m * i / G;
    it.rows = m * (i + 1) / G - it.row0;
    items[i] = it;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    *reinterpret_cast<int*>(scratch + kOffStatus) = 0;
    reinterpret_cast<int32_t*>(scratch + kOffItem0)[0] = 0;
    reinterpret_cast<int32_t*>(scratch + kOffItem0)[1] = G;
    *reinterpret_cast<float*>(scratch + kOffScale) = 1.0f / (float)m;
    *reinterpret_cast<int32_t*>(scratch + kOffDest) = 0;
  }
}

// Device address of g_scratch on the current device (looked up once).
int scratch_address(unsigned char** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PGC_ECUDA;
  if (dev < 0 || dev >= kMaxDevices) return PGC_ENOTSUP;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess || !p) return PGC_ECUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = static_cast<unsigned char*>(g_scratch_ptr[dev]);
  return PGC_OK;
}

}  // namespace

extern "C" int pgc_gradient_noalloc(int32_t loss, int32_t dtype, int64_t m, int64_t d, const void* X,
                                    const float* y, const float* w, float* g_out, void* stream) {
  if (loss != PGC_LOGISTIC && loss != PGC_LSQ) return PGC_EINVAL;
  if (dtype != PGC_F32 && dtype != PGC_BF16) return PGC_EINVAL;
  if (m < 1 || d < 1 || !X || !y || !w || !g_out) return PGC_EINVAL;
  if (reinterpret_cast<uintptr_t>(X) % 16 != 0 || reinterpret_cast<uintptr_t>(g_out) % 16 != 0)
    return PGC_EINVAL;
  int64_t ld = 0;
  const int variant = pgc::grad_rows_variant(dtype, d, &ld);
  if (variant < 0 || ld != d) return PGC_ENOTSUP;   // rows must need no padding

  unsigned char* scratch = nullptr;
  int rc = scratch_address(&scratch);
  if (rc) return rc;
  int sms = 148, dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return PGC_ECUDA;

  // one work item (one CTA) per SM, at least one stage of rows each
  const int64_t sr = pgc::grad_rows_stage_rows(variant, ld, dtype);
  int64_t G = std::min<int64_t>(sms, (m + sr - 1) / sr);
  G = std::max<int64_t>(G, 1);
  // the gradient kernel copies labels per stage from a 16-byte aligned start
  // and may read 12 bytes past the last one, so it reads a padded copy here
  const size_t off_labels = align256(kOffItems + (size_t)G * sizeof(pgc::WorkItem));
  const size_t off_partials = align256(off_labels + (size_t)m * sizeof(float) + 16);
  if (off_partials + (size_t)G * (size_t)ld * sizeof(float) > kScratchBytes) return PGC_ESCRATCH;

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  noalloc_fill_tables<<<(unsigned)((G + 255) / 256), 256, 0, st>>>(scratch, (int)G, m);
  if (cudaGetLastError() != cudaSuccess) return PGC_ECUDA;
  if (cudaMemcpyAsync(scratch + off_labels, y, (size_t)m * sizeof(float), cudaMemcpyDeviceToDevice, st) !=
      cudaSuccess)
    return PGC_ECUDA;

  pgc::GradRowsArgs g;
  g.loss = loss; g.dtype = dtype; g.d = d; g.ld = ld; g.X = X;
  g.y = reinterpret_cast<const float*>(scratch + off_labels); g.w = w;
  g.items = reinterpret_cast<const pgc::WorkItem*>(scratch + kOffItems);
  g.nitems = (int)G;
  int64_t max_rows = 0;
  for (int64_t i = 0; i < G; ++i) max_rows = std::max(max_rows, m * (i + 1) / G - m * i / G);
  g.max_item_rows = (int)max_rows;
  g.partials = reinterpret_cast<float*>(scratch + off_partials);
  g.status = reinterpret_cast<int*>(scratch + kOffStatus);
  if (pgc::launch_grad_rows(g, variant, st) != cudaSuccess) return PGC_ECUDA;

  pgc::CommitArgs c;
  c.partials = g.partials; c.P = ld;
  c.e_item0 = reinterpret_cast<const int32_t*>(scratch + kOffItem0);
  c.e_scale = reinterpret_cast<const float*>(scratch + kOffScale);
  c.e_dest = reinterpret_cast<const int32_t*>(scratch + kOffDest);
  c.ndest = 1; c.nE = 1; c.store = g_out;
  if (pgc::launch_commit(c, st) != cudaSuccess) return PGC_ECUDA;

  int status = 0;
  if (cudaMemcpyAsync(&status, scratch + kOffStatus, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return PGC_ECUDA;
  if (status & pgc::kErrWaitTimeout) return PGC_ETIMEOUT;
  return status ? PGC_ECUDA : PGC_OK;
}
