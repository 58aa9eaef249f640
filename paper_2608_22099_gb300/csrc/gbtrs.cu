// gbtrs.cu -- the solve after the factorisation: the backslash operator that the
// dispatch of Listing 1 stands for (Sec. I-A; LAPACK xGBTRS, no transpose).
//
// A X = B with A = P0 L0 P1 L1 ... U as left by gbtrf.  Each right-hand side is
// two chains of n dependent steps:
//   forward  j = 0..n-2: interchange b_j and b_{ipiv_j}; if b_j != 0, rows
//            j+1..j+kl take fma(-l, b_j, .);
//   backward j = n-1..0: if b_j != 0, b_j = b_j / u_jj and rows j-kv..j-1 take
//            fma(-b_j, u, .).
// One warp per right-hand side keeps the active part of b in registers, in a
// window that rotates with the steps (trwin.cuh); the division by u_jj uses a
// two-term reciprocal formed ahead of time, 32 diagonal entries at once
// (div_known: four dependent FP64 operations instead of a full division).  The
// same operations in the same order as the oracle, so the solution is
// bit-identical to it.  Interchanges outside j..j+kl (not produced by gbtrf)
// are ignored.
#include <climits>

#include "common.cuh"
#include "rcp.cuh"
#include "trwin.cuh"

namespace bandlu {
namespace {

// The two sweeps of a right-hand side (trwin.cuh), one warp each, as two
// kernels so that each gets its own window size and register allocation:
// forward with the interchanges and the multipliers (window >= kl+1), backward
// with U (window >= kl+ku+1).  kPf: steps read ahead.
template <int RW, int kPf>
__global__ void __launch_bounds__(128) k_gbtrs_fwd(int n, int kl, int ku, int nrhs, const double *__restrict__ AB,
                                                   int ldab, const int *__restrict__ ipiv, double *__restrict__ B,
                                                   long long ldb, const int *__restrict__ d_info) {
  const int rhs = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (rhs >= nrhs) return;  // whole warp
  if (d_info != nullptr && *d_info != 0) return;  // a singular factor: B is left as it is
  trwin::sweep<RW, kPf, true, true, false>(B + (long long)rhs * ldb, n, kl, trwin::GbLower{AB, ldab, kl + ku}, ipiv);
}

template <int RW, int kPf>
__global__ void __launch_bounds__(128) k_gbtrs_bwd(int n, int kl, int ku, int nrhs, const double *__restrict__ AB,
                                                   int ldab, double *__restrict__ B, long long ldb,
                                                   const int *__restrict__ d_info) {
  const int rhs = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (rhs >= nrhs) return;
  if (d_info != nullptr && *d_info != 0) return;
  const int kv = kl + ku;
  trwin::sweep<RW, kPf, false, false, true>(B + (long long)rhs * ldb, n, kv, trwin::GbUpper{AB, ldab, kv, n},
                                            nullptr);
}

// Any band: one warp per right-hand side, column by column through memory.
__global__ void __launch_bounds__(128) k_gbtrs_generic(int n, int kl, int ku, int nrhs, const double *__restrict__ AB,
                                                       long long ldab, const int *__restrict__ ipiv,
                                                       double *__restrict__ B, long long ldb,
                                                       const int *__restrict__ d_info) {
  const int lane = threadIdx.x & 31;
  const int rhs = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (rhs >= nrhs) return;
  if (d_info != nullptr && *d_info != 0) return;
  double *b = B + (long long)rhs * ldb;
  const long long kv = (long long)kl + ku;
  if (kl > 0) {
    for (int j = 0; j + 1 < n; ++j) {
      const int km = min(kl, n - 1 - j);
      const int l = ipiv[j] - 1;
      if (l != j && lane == 0) {
        const double t0 = b[l];
        b[l] = b[j];
        b[j] = t0;
      }
      __syncwarp();
      const double bj = b[j];
      if (nz(bj))
        for (int t = 1 + lane; t <= km; t += 32) b[j + t] = fma(-AB[(kv + t) + (long long)j * ldab], bj, b[j + t]);
      __syncwarp();
    }
  }
  for (int j = n - 1; j >= 0; --j) {
    double xj = b[j];
    if (nz(xj)) {
      xj = xj / AB[kv + (long long)j * ldab];
      const int i0 = (int)max(0LL, (long long)j - kv);
      for (int i = i0 + lane; i < j; i += 32) b[i] = fma(-xj, AB[(kv + i - j) + (long long)j * ldab], b[i]);
      __syncwarp();
      if (lane == 0) b[j] = xj;
    }
    __syncwarp();
  }
}

// Wide bands: one CTA per right-hand side.  The active part of b lives in a
// shared-memory ring of WS rows (a power of two >= kl+ku+1+32; row i in slot
// i mod WS).  Forward, the ring holds rows j..j+WS-1; backward, rows
// j-WS+1..j.  A step is one thread's interchange (or division), a barrier, the
// threads' updates of one row each, a barrier.  Every 32 steps the 32 slots of
// the rows just finished are refilled at once with the rows WS further on
// (needed no earlier than ku+1 steps later, so one load latency per 32 steps).
__global__ void __launch_bounds__(256) k_gbtrs_cta(int n, int kl, int ku, int WS, const double *__restrict__ AB,
                                                   long long ldab, const int *__restrict__ ipiv,
                                                   double *__restrict__ B, long long ldb,
                                                   const int *__restrict__ d_info) {
  extern __shared__ double ring[];  // WS
  const int tid = threadIdx.x, nt = blockDim.x;
  const int rhs = blockIdx.x;
  if (d_info != nullptr && *d_info != 0) return;
  double *b = B + (long long)rhs * ldb;
  const long long kv = (long long)kl + ku;
  const int mask = WS - 1;
  if (kl > 0 && n > 1) {
    for (int i = tid; i < WS; i += nt) ring[i] = i < n ? b[i] : 0.0;
    __syncthreads();
    for (int j = 0; j + 1 < n; ++j) {
      const int km = min(kl, n - 1 - j);
      if (j >= 32 && (j & 31) == 0 && tid < 32) {  // rows j-32..j-1 are final
        const int r = j - 32 + tid;
        ring[r & mask] = (r + WS < n) ? b[r + WS] : 0.0;
      }
      if (tid == 0) {
        const int l = ipiv[j] - 1;
        if (l != j) {
          const double t0 = ring[l & mask];
          ring[l & mask] = ring[j & mask];
          ring[j & mask] = t0;
        }
      }
      __syncthreads();
      const double bj = ring[j & mask];
      if (nz(bj))
        for (int t = 1 + tid; t <= km; t += nt)
          ring[(j + t) & mask] = fma(-AB[(kv + t) + (long long)j * ldab], bj, ring[(j + t) & mask]);
      if (tid == 0) b[j] = bj;  // y_j
      __syncthreads();
    }
    if (tid == 0) b[n - 1] = ring[(n - 1) & mask];
    __syncthreads();
  }
  for (int t = tid; t < WS; t += nt) {
    const int i = n - 1 - t;
    if (i >= 0) ring[i & mask] = b[i];
  }
  __syncthreads();
  for (int j = n - 1; j >= 0; --j) {
    const int done = n - 1 - j;  // rows j+1..n-1 are final
    if (done >= 32 && (done & 31) == 0 && tid < 32) {
      const int r = j + 1 + tid;  // rows j+1..j+32
      ring[r & mask] = (r - WS >= 0) ? b[r - WS] : 0.0;
    }
    double xj = ring[j & mask];
    if (nz(xj)) {  // uniform
      xj = xj / AB[kv + (long long)j * ldab];
      const int lo = (int)max(0LL, (long long)j - kv);
      for (int i = j - 1 - tid; i >= lo; i -= nt)
        ring[i & mask] = fma(-xj, AB[(kv + i - j) + (long long)j * ldab], ring[i & mask]);
    }
    if (tid == 0) b[j] = xj;
    __syncthreads();
  }
}

// read-ahead depth for a window of 32*RW rows: kPf steps must outlast a DRAM
// round trip (~2000 clocks)
template <int RW>
constexpr int pf_for() {
  return RW <= 2 ? 16 : (RW <= 8 ? 8 : 4);
}

template <int RW>
void launch_fwd(int n, int kl, int ku, int nrhs, const double *AB, int ldab, const int *ipiv, double *B, long long ldb,
                const int *d_info, cudaStream_t s) {
  const int wpb = 4;
  k_gbtrs_fwd<RW, pf_for<RW>()><<<(unsigned)((nrhs + wpb - 1) / wpb), 32 * wpb, 0, s>>>(n, kl, ku, nrhs, AB, ldab,
                                                                                      ipiv, B, ldb, d_info);
}

template <int RW>
void launch_bwd(int n, int kl, int ku, int nrhs, const double *AB, int ldab, double *B, long long ldb,
                const int *d_info, cudaStream_t s) {
  const int wpb = 4;
  k_gbtrs_bwd<RW, pf_for<RW>()><<<(unsigned)((nrhs + wpb - 1) / wpb), 32 * wpb, 0, s>>>(n, kl, ku, nrhs, AB, ldab,
                                                                                      B, ldb, d_info);
}

// Register windows for both sweeps (kl+ku+1 <= 512).
int launch_window(int n, int kl, int ku, int nrhs, const double *AB, int ldab, const int *ipiv, double *B,
                  long long ldb, const int *d_info, cudaStream_t s) {
  if (kl > 0 && n > 1) {
    const int wf = kl + 1;
    if (wf <= 32) launch_fwd<1>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    else if (wf <= 64) launch_fwd<2>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    else if (wf <= 128) launch_fwd<4>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    else if (wf <= 256) launch_fwd<8>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    else launch_fwd<16>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    BANDLU_CHECK_LAUNCH();
  }
  const int wb = kl + ku + 1;
  if (wb <= 32) launch_bwd<1>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  else if (wb <= 64) launch_bwd<2>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  else if (wb <= 128) launch_bwd<4>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  else if (wb <= 256) launch_bwd<8>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  else launch_bwd<16>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace

int launch_gbtrs(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
                 int64_t ldb, const int *d_info, cudaStream_t s) {
  if (n == 0 || nrhs == 0) return BANDLU_OK;
  const long long win = (long long)kl + ku + 1;  // rows the backward window needs (>= kl + 1)
  if (n <= INT_MAX / 2 && ldab <= INT_MAX && nrhs <= INT_MAX) {
    if (win <= 512) return launch_window((int)n, kl, ku, (int)nrhs, AB, (int)ldab, ipiv, B, ldb, d_info, s);
  }
  // wider bands: a CTA per right-hand side with a shared-memory ring
  int WS = 1;
  while (WS < win + 32) WS <<= 1;
  if (n <= INT_MAX / 2 && nrhs <= INT_MAX && (size_t)WS * sizeof(double) <= 96 * 1024) {
    if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_gbtrs_cta), 96 * 1024)) return BANDLU_ERR_CUDA;
    k_gbtrs_cta<<<(unsigned)nrhs, 256, (size_t)WS * sizeof(double), s>>>((int)n, kl, ku, WS, AB, ldab, ipiv, B, ldb,
                                                                        d_info);
    BANDLU_CHECK_LAUNCH();
    return BANDLU_OK;
  }
  const int wpb = 4;
  const long long grid = (nrhs + wpb - 1) / wpb;
  k_gbtrs_generic<<<(unsigned)grid, 32 * wpb, 0, s>>>((int)n, kl, ku, (int)nrhs, AB, ldab, ipiv, B, ldb, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu
