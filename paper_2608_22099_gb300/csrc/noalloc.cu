// noalloc.cu -- dispatch_lu_noalloc: dispatch_lu without any device allocation.
//
// dispatch_lu takes 8 bytes of device scratch per call for the detected (kl, ku)
// from the stream-ordered allocator.  Some callers cannot allocate device memory
// from inside a library call: a process whose device memory is entirely reserved
// by its own caching allocator (an extra cudaMallocAsync can fail or fragment the
// pool), or a latency-critical loop whose rules forbid allocation calls, which can
// take driver locks or synchronize.  This entry point keeps that scratch in a
// file-scope __device__ array instead; every GPU that loads the library holds the
// array (kNoAllocScratchBytes) until the process exits.
#include <cuda.h>

#include <mutex>

#include "common.cuh"

namespace {

// Scratch of dispatch_lu_noalloc: element 0 = kl, element 1 = ku of the current call.
// Every call shares it and it keeps the last call's values; the detection launch
// clears both elements before it folds in the new bandwidths.
static __device__ __align__(256) int g_noalloc_scratch[64];
constexpr size_t kNoAllocScratchBytes = sizeof(int) * 64;
constexpr size_t kNoAllocScratchNeeded = 2 * sizeof(int);  // what one call uses, for every n
constexpr int kMaxDevices = 64;

// The array's device address is looked up once per device context: a reset of the
// device (cudaDeviceReset) ends the context, its module and the array with it, and the
// next call on that device looks the address up again in the new context.  Contexts are
// told apart by the driver's unique context id (cuCtxGetId), reached through the
// runtime's driver entry points so the library needs no link to the driver library.
typedef CUresult (*PFN_ctxGetCurrent)(CUcontext *);
typedef CUresult (*PFN_ctxGetId)(CUcontext, unsigned long long *);

struct ScratchCache {
  int *ptr = nullptr;
  unsigned long long ctx_id = 0;
};

std::mutex g_setup_mu;
ScratchCache g_cache[kMaxDevices];
bool g_entry_points_tried = false;
PFN_ctxGetCurrent g_ctx_get_current = nullptr;
PFN_ctxGetId g_ctx_get_id = nullptr;

// Id of the current device's context, or 0 when the driver cannot report one.
unsigned long long current_context_id() {
  if (!g_entry_points_tried) {
    g_entry_points_tried = true;
    cudaDriverEntryPointQueryResult q;
    void *f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_ctx_get_current = reinterpret_cast<PFN_ctxGetCurrent>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_ctx_get_id = reinterpret_cast<PFN_ctxGetId>(f);
  }
  if (g_ctx_get_current == nullptr || g_ctx_get_id == nullptr) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (g_ctx_get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
  if (g_ctx_get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of the scratch array on the current device, resolved with that
// device current, once per device context (always, when the context id is not
// available).  Returns nullptr and sets *err on failure.
int *scratch_for_current_device(int *err) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *err = BANDLU_ERR_CUDA;
    return nullptr;
  }
  // makes the device's primary context current (initialising it if needed), so the
  // context id below is the one the launches of this call will run in
  if (cudaSetDevice(dev) != cudaSuccess) {
    *err = BANDLU_ERR_CUDA;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_setup_mu);
  const unsigned long long id = current_context_id();
  ScratchCache &c = g_cache[dev];
  if (c.ptr == nullptr || id == 0 || c.ctx_id != id) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
      *err = BANDLU_ERR_CUDA;
      return nullptr;
    }
    c.ptr = static_cast<int *>(p);
    c.ctx_id = id;
  }
  return c.ptr;
}

}  // namespace

extern "C" int dispatch_lu_noalloc(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv,
                                   int *h_kl, int *h_ku, int *d_info, cudaStream_t stream) {
  if (A == nullptr && n > 0) return -1;
  if (n < 0 || n > (int64_t)INT32_MAX) return -2;
  const int64_t n1 = n > 1 ? n : 1;
  if (lda < n1 || lda > INT64_MAX / n1) return -3;
  if (AB == nullptr && n > 0) return -4;
  if (ldab < 1 || ldab > INT64_MAX / n1) return -5;
  if (ipiv == nullptr && n > 0) return -6;
  if (h_kl == nullptr) return -7;
  if (h_ku == nullptr) return -8;
  if (d_info == nullptr) return -9;
  if (kNoAllocScratchNeeded > kNoAllocScratchBytes) return BANDLU_ERR_SCRATCH;
  int err = BANDLU_OK;
  int *scratch = scratch_for_current_device(&err);
  if (scratch == nullptr) return err;
  int rc = bandlu::launch_detect(A, n, lda, scratch, scratch + 1, stream);
  int h[2] = {0, 0};
  if (rc == BANDLU_OK && cudaMemcpyAsync(h, scratch, sizeof(h), cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    rc = BANDLU_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (rc != BANDLU_OK) return rc;
  *h_kl = h[0];
  *h_ku = h[1];
  if (!bandlu::predicate_banded(n, h[0], h[1], ldab)) return BANDLU_NOT_BANDED;
  rc = bandlu::launch_dense_to_band(A, lda, n, h[0], h[1], AB, ldab, stream);
  if (rc != BANDLU_OK) return rc;
  return bandlu::launch_gbtrf(n, h[0], h[1], AB, ldab, ipiv, d_info, stream, /*allow_alloc=*/false);
}
