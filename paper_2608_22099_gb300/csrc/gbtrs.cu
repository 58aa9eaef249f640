// gbtrs.cu -- the solve after the factorisation: the backslash operator that the
// dispatch of Listing 1 stands for (Sec. I-A; LAPACK xGBTRS, no transpose).
//
// A X = B with A = P0 L0 P1 L1 ... U as left by gbtrf.  Each right-hand side is
// two chains of n dependent steps:
//   forward  j = 0..n-2: interchange b_j and b_{ipiv_j}; if b_j != 0, rows
//            j+1..j+kl take fma(-l, b_j, .);
//   backward j = n-1..0: if b_j != 0, b_j = b_j / u_jj and rows j-kv..j-1 take
//            fma(-b_j, u, .).
// One warp per right-hand side keeps the active part of b in registers (a
// window of W = 32*RW rows: row t of the window on lane t % 32, register t / 32),
// reads each step's factor column kPf steps ahead (the step loop is unrolled by
// kPf so that every prefetch slot is one register), and writes every finished
// entry once.  The same operations in the same order as the oracle, so the
// solution is bit-identical to it.
#include <climits>

#include "common.cuh"

namespace bandlu {
namespace {

constexpr int kPf = 4;  // steps read ahead

// Element t of the window (t warp-uniform).
template <int RW>
__device__ __forceinline__ double win_get(const double (&w)[RW], int t) {
  double v = 0.0;
#pragma unroll
  for (int r = 0; r < RW; ++r) {
    const double x = __shfl_sync(FULL, w[r], t & 31);
    if (r == (t >> 5)) v = x;
  }
  return v;
}

template <int RW>
__device__ __forceinline__ void win_set(double (&w)[RW], int t, double v, int lane) {
#pragma unroll
  for (int r = 0; r < RW; ++r)
    if (r == (t >> 5) && lane == (t & 31)) w[r] = v;
}

// w[t] = w[t+1] for every t; the last row takes `in`.
template <int RW>
__device__ __forceinline__ void win_shift(double (&w)[RW], double in, int lane) {
#pragma unroll
  for (int r = 0; r < RW; ++r) {
    const double carry = (r + 1 < RW) ? __shfl_sync(FULL, w[r + 1 < RW ? r + 1 : r], 0) : in;
    const double sh = __shfl_down_sync(FULL, w[r], 1);
    w[r] = lane == 31 ? carry : sh;
  }
}

template <int RW>
__global__ void __launch_bounds__(128) k_gbtrs_window(int n, int kl, int ku, int nrhs, const double *__restrict__ AB,
                                                      int ldab, const int *__restrict__ ipiv, double *__restrict__ B,
                                                      long long ldb, const int *__restrict__ d_info) {
  constexpr int W = 32 * RW;
  const int lane = threadIdx.x & 31;
  const int rhs = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (rhs >= nrhs) return;  // whole warp
  if (d_info != nullptr && *d_info != 0) return;  // a singular factor: B is left as it is
  double *b = B + (long long)rhs * ldb;
  const int kv = kl + ku;

  // ---------------- forward: window row t = b_{j+t} ----------------
  if (kl > 0 && n > 1) {
    double w[RW];
#pragma unroll
    for (int r = 0; r < RW; ++r) {
      const int t = lane + 32 * r;
      w[r] = t < n ? b[t] : 0.0;
    }
    // slot s: multipliers of step j = j0 + s (window row t = 1..kl) and the row
    // entering the window after it (b_{j+W})
    double lm[kPf][RW], en[kPf];
    int pv[kPf];
#pragma unroll
    for (int s = 0; s < kPf; ++s) {
      const int j = s;
#pragma unroll
      for (int r = 0; r < RW; ++r) {
        const int t = lane + 32 * r;
        lm[s][r] = (j < n - 1 && t >= 1 && t <= min(kl, n - 1 - j)) ? AB[(kv + t) + (long long)j * ldab] : 0.0;
      }
      en[s] = (lane == 31 && j + W < n) ? b[j + W] : 0.0;
      pv[s] = j < n - 1 ? ipiv[j] - 1 - j : 0;
    }
    for (int j0 = 0; j0 < n - 1; j0 += kPf) {
#pragma unroll
      for (int s = 0; s < kPf; ++s) {
        const int j = j0 + s;
        if (j >= n - 1) break;
        const int km = min(kl, n - 1 - j);
        const int p = pv[s];
        if (p != 0) {  // uniform
          const double a = win_get(w, 0), c = win_get(w, p);
          win_set(w, 0, c, lane);
          win_set(w, p, a, lane);
        }
        const double bj = win_get(w, 0);
        if (lane == 0) b[j] = bj;  // y_j
        if (nz(bj)) {
#pragma unroll
          for (int r = 0; r < RW; ++r) {
            const int t = lane + 32 * r;
            if (t >= 1 && t <= km) w[r] = fma(-lm[s][r], bj, w[r]);
          }
        }
        win_shift(w, en[s], lane);
        // refill the slot with step j + kPf
        const int jn = j + kPf;
#pragma unroll
        for (int r = 0; r < RW; ++r) {
          const int t = lane + 32 * r;
          lm[s][r] = (jn < n - 1 && t >= 1 && t <= min(kl, n - 1 - jn)) ? AB[(kv + t) + (long long)jn * ldab] : 0.0;
        }
        en[s] = (lane == 31 && jn + W < n) ? b[jn + W] : 0.0;
        pv[s] = jn < n - 1 ? ipiv[jn] - 1 - jn : 0;
      }
    }
    const double last = win_get(w, 0);
    if (lane == 0) b[n - 1] = last;
    __syncwarp();  // the backward sweep reads what other lanes wrote
  }

  // ---------------- backward: window row t = b_{j-t} ----------------
  {
    double w[RW];
#pragma unroll
    for (int r = 0; r < RW; ++r) {
      const int t = lane + 32 * r;
      w[r] = t <= n - 1 ? b[n - 1 - t] : 0.0;
    }
    // slot s: column j = n-1-(j0+s) of U (window row t <-> U(j-t, j) = AB(kv-t, j))
    // and the row entering after it (b_{j-W})
    double uc[kPf][RW], en[kPf];
#pragma unroll
    for (int s = 0; s < kPf; ++s) {
      const int j = n - 1 - s;
#pragma unroll
      for (int r = 0; r < RW; ++r) {
        const int t = lane + 32 * r;
        uc[s][r] = (j >= 0 && t <= min(kv, j)) ? AB[(kv - t) + (long long)j * ldab] : 0.0;
      }
      en[s] = (lane == 31 && j - W >= 0) ? b[j - W] : 0.0;
    }
    for (int i0 = 0; i0 < n; i0 += kPf) {
#pragma unroll
      for (int s = 0; s < kPf; ++s) {
        const int j = n - 1 - (i0 + s);
        if (j < 0) break;
        double xj = win_get(w, 0);
        if (nz(xj)) {  // uniform
          xj = xj / __shfl_sync(FULL, uc[s][0], 0);  // u_jj
#pragma unroll
          for (int r = 0; r < RW; ++r) {
            const int t = lane + 32 * r;
            if (t >= 1 && t <= min(kv, j)) w[r] = fma(-xj, uc[s][r], w[r]);
          }
        }
        if (lane == 0) b[j] = xj;  // x_j (a zero entry stays as the updates left it)
        win_shift(w, en[s], lane);
        const int jn = j - kPf;
#pragma unroll
        for (int r = 0; r < RW; ++r) {
          const int t = lane + 32 * r;
          uc[s][r] = (jn >= 0 && t <= min(kv, jn)) ? AB[(kv - t) + (long long)jn * ldab] : 0.0;
        }
        en[s] = (lane == 31 && jn - W >= 0) ? b[jn - W] : 0.0;
      }
    }
  }
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

template <int RW>
int launch_rw(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
              int64_t ldb, const int *d_info, cudaStream_t s) {
  const int wpb = 4;
  const long long grid = (nrhs + wpb - 1) / wpb;
  k_gbtrs_window<RW><<<(unsigned)grid, 32 * wpb, 0, s>>>((int)n, kl, ku, (int)nrhs, AB, (int)ldab, ipiv, B, ldb,
                                                         d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace

int launch_gbtrs(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
                 int64_t ldb, const int *d_info, cudaStream_t s) {
  if (n == 0 || nrhs == 0) return BANDLU_OK;
  const long long win = (long long)kl + ku + 1;  // rows the backward window needs (>= kl + 1)
  if (n <= INT_MAX / 2 && ldab <= INT_MAX && nrhs <= INT_MAX) {
    if (win <= 32) return launch_rw<1>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    if (win <= 64) return launch_rw<2>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    if (win <= 128) return launch_rw<4>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    if (win <= 256) return launch_rw<8>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    if (win <= 512) return launch_rw<16>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
  }
  // wider bands: a CTA per right-hand side with a shared-memory ring
  int WS = 1;
  while (WS < win + 32) WS <<= 1;
  if (n <= INT_MAX / 2 && nrhs <= INT_MAX && (size_t)WS * sizeof(double) <= 96 * 1024) {
    static bool attr = false;
    if (!attr) {
      if (cudaFuncSetAttribute(k_gbtrs_cta, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024) != cudaSuccess)
        return BANDLU_ERR_CUDA;
      attr = true;
    }
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
