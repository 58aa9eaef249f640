// common.cuh -- shared device helpers of the banded LU library (sm_103a).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "bandlu.h"

namespace bandlu {

constexpr unsigned FULL = 0xffffffffu;

// IEEE "a != 0.0" on the bit pattern: true for every value except +0.0 and -0.0
// (NaN, +-Inf and subnormals are nonzero).  Integer-only, so it never issues on
// the FP64 pipe.
__device__ __forceinline__ bool nz_bits(unsigned long long b) { return (b << 1) != 0ull; }
// The same test on a double, done on its two 32-bit halves: the 64-bit form of
// a double's bits can be compiled back into a floating-point compare, which
// issues on the FP64 pipe at the FMA rate.
__device__ __forceinline__ bool nz(double x) {
  return ((((unsigned)__double2hiint(x)) << 1) | (unsigned)__double2loint(x)) != 0u;
}

// c ? a : b as one PTX select of the 64-bit patterns.  Register windows pick
// their rows with it: a chain of plain selects on a runtime row index can be
// turned by the compiler into an indexed array in local memory, which puts a
// local load on every step's dependence chain.
__device__ __forceinline__ double dsel(bool c, double a, double b) {
  unsigned long long r;
  asm("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %3, 0;\n\tselp.b64 %0, %1, %2, q;\n\t}"
      : "=l"(r)
      : "l"((unsigned long long)__double_as_longlong(a)), "l"((unsigned long long)__double_as_longlong(b)),
        "r"((unsigned)c));
  return __longlong_as_double((long long)r);
}

// Pivot-search key of a candidate: for non-NaN doubles |x| < |y| iff
// key(x) < key(y).  The xGBTRF comparison order starts its running best at the
// first candidate and replaces it only by a strictly larger modulus, which a
// NaN never is: so a NaN gets the largest key as the first candidate (it is
// kept) and the key of zero otherwise (with the first-index rule on ties it is
// never chosen over an earlier candidate).
__device__ __forceinline__ unsigned long long pivot_abs_key(double x, bool first) {
  const unsigned hi = (unsigned)__double2hiint(x) & 0x7fffffffu, lo = (unsigned)__double2loint(x);
  const bool nan = hi > 0x7ff00000u || (hi == 0x7ff00000u && lo != 0u);
  return nan ? (first ? ~0ull : 0ull) : (((unsigned long long)hi << 32) | lo);
}

// First lane holding the largest key among all 32 lanes (ties -> lowest lane).
// Exact on 63-bit keys using two 32-bit max reductions and a ballot.
__device__ __forceinline__ int warp_argmax_first(unsigned long long key) {
  const unsigned hi = (unsigned)(key >> 32), lo = (unsigned)key;
  const unsigned mhi = __reduce_max_sync(FULL, hi);
  const unsigned lo2 = (hi == mhi) ? lo : 0u;
  const unsigned mlo = __reduce_max_sync(FULL, lo2);
  const unsigned win = __ballot_sync(FULL, hi == mhi && lo == mlo);
  return __ffs(win) - 1;
}

// As warp_argmax_first, and *all_zero tells whether every key is zero.  When
// one lane alone holds the largest high word (the usual case) it is the
// winner and the reduction over the low words is skipped.
__device__ __forceinline__ int warp_argmax_first_z(unsigned long long key, bool *all_zero) {
  const unsigned hi = (unsigned)(key >> 32), lo = (unsigned)key;
  const unsigned mhi = __reduce_max_sync(FULL, hi);
  const unsigned top = __ballot_sync(FULL, hi == mhi);
  if (__popc(top) == 1) {  // uniform; then mhi > 0 (mhi == 0 would put every lane in top)
    *all_zero = false;
    return __ffs(top) - 1;
  }
  const unsigned lo2 = (hi == mhi) ? lo : 0u;
  const unsigned mlo = __reduce_max_sync(FULL, lo2);
  const unsigned win = __ballot_sync(FULL, hi == mhi && lo == mlo);
  *all_zero = (mhi | mlo) == 0u;
  return __ffs(win) - 1;
}

// (key, index) pair that prefers the larger key and, on a tie, the smaller index.
struct KeyIdx {
  unsigned long long key;
  long long idx;
};
__device__ __forceinline__ KeyIdx better(KeyIdx a, KeyIdx b) {
  if (b.key > a.key || (b.key == a.key && b.idx < a.idx)) return b;
  return a;
}
__device__ __forceinline__ KeyIdx warp_reduce_keyidx(KeyIdx v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    KeyIdx o;
    o.key = __shfl_xor_sync(FULL, v.key, off);
    o.idx = __shfl_xor_sync(FULL, v.idx, off);
    v = better(v, o);
  }
  return v;
}

// Dispatch predicate (Eq. su-con with integer operation counts, and the storage
// capacity): banded iff 3*(n^2 + n*(kl+ku+1) + n*kl*(2*(kl+ku)+1)) < 2*n^3 and
// 2*kl+ku+1 <= ldab.  128-bit arithmetic: exact for every n < 2^31.
__host__ __device__ inline bool predicate_banded(long long n, long long kl, long long ku, long long ldab) {
  if (2 * kl + ku + 1 > ldab) return false;
  const __int128 N = n, L = kl, U = ku;
  const __int128 lhs = 3 * (N * N + N * (L + U + 1) + N * L * (2 * (L + U) + 1));
  return lhs < 2 * N * N * N;
}

// The cluster-pair wide factorisation takes a band (whose window factorisation
// path is the generic one) when its panels of kl + 4 rows fit the compute group of
// `rows_cap` threads the kernel was launched with (0: not launched) and the band
// spans at least two 4-column blocks (n >= 16, kl >= 1, kl + ku >= 8).  The
// device-side dispatch and the kernel both apply this rule.
__host__ __device__ inline bool wide_pair_takes(long long n, int kl, int ku, int rows_cap) {
  return rows_cap > 0 && n >= 16 && kl >= 1 && (long long)kl + ku >= 8 && kl + 4 <= rows_cap;
}

}  // namespace bandlu

#define BANDLU_CHECK_LAUNCH()                         \
  do {                                                \
    if (cudaPeekAtLastError() != cudaSuccess) return BANDLU_ERR_CUDA; \
  } while (0)

// Launchers shared between the C-ABI translation unit and the kernel units.
namespace bandlu {
// Opts `kernel` in to `bytes` of dynamic shared memory on the current device,
// once per (kernel, device) pair; thread-safe.  Returns false if CUDA refuses.
bool allow_dynamic_smem(const void *kernel, int bytes);
// Number of SMs of the current device (looked up once per device; thread-safe).
int device_sms();
int launch_detect(const double *A, int64_t n, int64_t lda, int *d_kl, int *d_ku, cudaStream_t s);
int launch_dense_to_band(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                         cudaStream_t s);
// Column-major input, A(i,j) = A[i + j*lda].
int launch_dense_to_band_cm(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                            cudaStream_t s);
// allow_alloc = false keeps the launch free of device allocations (wide bands
// then take the single-CTA kernel instead of the multi-CTA one, whose
// hand-off flags live in stream-ordered scratch).
int launch_gbtrf(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t s,
                 bool allow_alloc = true);
int launch_gbtrf_wide(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t s,
                      bool *used);
// dispatch_lu_async: the decision and the conversion with (kl, ku) read on the
// device (*d_status = BANDLU_OK or BANDLU_NOT_BANDED), then the factorisation
// it selects (nothing when declined).
int launch_decide_convert(const double *A, int64_t lda, int64_t n, int64_t ldab, const int *d_kl, const int *d_ku,
                          int *d_status, double *AB, cudaStream_t s);
int launch_gbtrf_on_device(int64_t n, double *AB, int64_t ldab, int *ipiv, const int *d_kl, const int *d_ku,
                           const int *d_status, int *d_info, cudaStream_t s);
// dispatch_lu_async's wide path: the cluster-pair kernel enqueued with the band
// storage's largest admissible kl ((ldab-1)/2) before (kl, ku) are known.
// prepare: when that kernel can be made resident for this ldab, takes and clears
// its hand-off flags (stream-ordered) and sets *rows_cap > 0 and *flags; else
// *rows_cap = 0.  launch: enqueues the kernel (which reads (kl, ku) and the
// decision flags[1] on the device and exits unless the band is its) and frees the
// flags.
struct WideDeferred {
  int rows_cap = 0;
  int cw = 0;
  bool chain = false;  // the streaming chain kernel (else the cluster pair)
  int grid = 0;
  size_t smem = 0;
  int *flags = nullptr;
};
int prepare_gbtrf_wide_deferred(int64_t n, int64_t ldab, cudaStream_t s, WideDeferred *wd);
int launch_gbtrf_wide_deferred(const WideDeferred &wd, int64_t n, double *AB, int64_t ldab, int *ipiv,
                               const int *d_kl, const int *d_ku, int *d_info, cudaStream_t s);
// d_info: when not null and *d_info != 0 (a singular factor), B is left as it is.
int launch_gbtrs(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
                 int64_t ldb, const int *d_info, cudaStream_t s);
// Triangular solve with the band of width k of A's lower (or upper) triangle,
// and the diagonal solve; both write *d_info (first zero diagonal entry).
int launch_trsv(bool lower, int64_t n, int k, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs,
                int *d_info, cudaStream_t s);
int launch_diag_solve(int64_t n, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs, int *d_info,
                      cudaStream_t s);
int launch_batched(const double *A, int64_t n, int64_t lda, int64_t strideA, int64_t batch, double *AB,
                   int64_t ldab, int64_t strideAB, int *ipiv, int64_t strideP, int *d_kl, int *d_ku, int *d_info,
                   int *d_status, cudaStream_t s);
}  // namespace bandlu
