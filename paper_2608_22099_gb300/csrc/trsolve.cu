// trsolve.cu -- the triangular and diagonal branches of the backslash dispatch
// (Listing 1, Sec. I-A): solves with a triangle of bandwidth k read in place
// from the dense row-major matrix (no format conversion: the band's entries of
// column j are A(j+t, j), one row apart), and the diagonal solve.
//
//  * k_first_zero_diag: the xTRTRS singularity check, info = first i with
//    A(i,i) == 0 (1-based) or 0; the solves read it on the device and leave B
//    as it is when it is nonzero.
//  * k_trsv_window<RW, kPf, kLower>: one warp per right-hand side, a register
//    window of the right-hand side (trwin.cuh) for k + 1 <= 512: the
//    column-oriented substitution of xTBSV with the reference BLAS's zero test
//    and the IEEE quotient (div_known); each row's band segment is asked of L2
//    ahead of its first use (trwin's DenseLower / DenseUpper sources).
//  * k_trsv_generic: any k, one warp per right-hand side through memory.
//  * k_diag_solve: B(i,c) / A(i,i) for every entry, one thread each.
#include <climits>

#include "common.cuh"
#include "trwin.cuh"

namespace bandlu {
namespace {

__global__ void __launch_bounds__(1024) k_first_zero_diag(const double *__restrict__ A, long long lda, long long n,
                                                          int *__restrict__ d_info) {
  __shared__ long long s_min[32];
  long long first = LLONG_MAX;
  for (long long i = threadIdx.x; i < n; i += blockDim.x) {
    if (!nz(A[i * lda + i])) {
      first = i;
      break;  // later i of this thread are larger
    }
  }
  for (int off = 16; off > 0; off >>= 1) first = min(first, __shfl_xor_sync(FULL, first, off));
  if ((threadIdx.x & 31) == 0) s_min[threadIdx.x >> 5] = first;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long m = LLONG_MAX;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = min(m, s_min[w]);
    *d_info = m == LLONG_MAX ? 0 : (int)(m + 1);
  }
}

template <int RW, int kPf, bool kLower>
__global__ void __launch_bounds__(128) k_trsv_window(int n, int k, const double *__restrict__ A, long long lda,
                                                     double *__restrict__ B, long long ldb, int nrhs,
                                                     const int *__restrict__ d_info) {
  const int rhs = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (rhs >= nrhs) return;  // whole warp
  if (*d_info != 0) return;  // a zero on the diagonal: B is left as it is
  double *b = B + (long long)rhs * ldb;
  if (kLower)
    trwin::sweep<RW, kPf, true, false, true>(b, n, k, trwin::DenseLower{A, lda}, nullptr);
  else
    trwin::sweep<RW, kPf, false, false, true>(b, n, k, trwin::DenseUpper{A, lda, n}, nullptr);
}

__global__ void __launch_bounds__(128) k_trsv_generic(int lower, long long n, long long k, const double *__restrict__ A,
                                                      long long lda, double *__restrict__ B, long long ldb,
                                                      long long nrhs, const int *__restrict__ d_info) {
  const int lane = threadIdx.x & 31;
  const long long rhs = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (rhs >= nrhs) return;
  if (*d_info != 0) return;
  double *b = B + rhs * ldb;
  for (long long s = 0; s < n; ++s) {
    const long long j = lower ? s : n - 1 - s;
    double xj = b[j];
    if (nz(xj)) {  // uniform
      xj = xj / A[j * lda + j];
      const long long i0 = lower ? j + 1 : max(0LL, j - k), i1 = lower ? min(n - 1, j + k) : j - 1;
      for (long long i = i0 + lane; i <= i1; i += 32) b[i] = fma(-xj, A[i * lda + j], b[i]);
      __syncwarp();
      if (lane == 0) b[j] = xj;
    }
    __syncwarp();
  }
}

__global__ void k_diag_solve(long long n, const double *__restrict__ A, long long lda, double *__restrict__ B,
                             long long ldb, long long nrhs, const int *__restrict__ d_info) {
  if (*d_info != 0) return;
  const long long total = n * nrhs;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const long long c = e / n, i = e - c * n;
    B[c * ldb + i] = B[c * ldb + i] / A[i * lda + i];
  }
}

template <int RW, bool kLower>
int launch_trsv_rw(int n, int k, const double *A, long long lda, double *B, long long ldb, int nrhs,
                   const int *d_info, cudaStream_t s) {
  constexpr int kPf = RW <= 2 ? 16 : (RW <= 8 ? 8 : 4);
  const int wpb = 4;
  k_trsv_window<RW, kPf, kLower><<<(unsigned)((nrhs + wpb - 1) / wpb), 32 * wpb, 0, s>>>(n, k, A, lda, B, ldb,
                                                                                         nrhs, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

template <bool kLower>
int launch_trsv_window(int n, int k, const double *A, long long lda, double *B, long long ldb, int nrhs,
                       const int *d_info, cudaStream_t s) {
  const int w = k + 1;
  if (w <= 32) return launch_trsv_rw<1, kLower>(n, k, A, lda, B, ldb, nrhs, d_info, s);
  if (w <= 64) return launch_trsv_rw<2, kLower>(n, k, A, lda, B, ldb, nrhs, d_info, s);
  if (w <= 128) return launch_trsv_rw<4, kLower>(n, k, A, lda, B, ldb, nrhs, d_info, s);
  if (w <= 256) return launch_trsv_rw<8, kLower>(n, k, A, lda, B, ldb, nrhs, d_info, s);
  return launch_trsv_rw<16, kLower>(n, k, A, lda, B, ldb, nrhs, d_info, s);
}

int launch_first_zero_diag(const double *A, int64_t lda, int64_t n, int *d_info, cudaStream_t s) {
  k_first_zero_diag<<<1, 1024, 0, s>>>(A, lda, n, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace

int launch_trsv(bool lower, int64_t n, int k, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs,
                int *d_info, cudaStream_t s) {
  int rc = launch_first_zero_diag(A, lda, n, d_info, s);
  if (rc != BANDLU_OK || n == 0 || nrhs == 0) return rc;
  if (k + 1 <= 512 && n <= INT_MAX / 2 && nrhs <= INT_MAX) {
    return lower ? launch_trsv_window<true>((int)n, k, A, lda, B, ldb, (int)nrhs, d_info, s)
                 : launch_trsv_window<false>((int)n, k, A, lda, B, ldb, (int)nrhs, d_info, s);
  }
  const int wpb = 4;
  k_trsv_generic<<<(unsigned)((nrhs + wpb - 1) / wpb), 32 * wpb, 0, s>>>(lower ? 1 : 0, n, k, A, lda, B, ldb, nrhs,
                                                                         d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

int launch_diag_solve(int64_t n, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs, int *d_info,
                      cudaStream_t s) {
  int rc = launch_first_zero_diag(A, lda, n, d_info, s);
  if (rc != BANDLU_OK || n == 0 || nrhs == 0) return rc;
  long long blocks = (n * nrhs + 255) / 256;
  if (blocks > 152ll * 32) blocks = 152ll * 32;
  k_diag_solve<<<(unsigned)blocks, 256, 0, s>>>(n, A, lda, B, ldb, nrhs, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu
