// batched.cu -- the strategy of Sec. II-A over a batch of independent matrices,
// with no host round trip: every matrix gets its own identification, decision,
// conversion and factorisation.
//
//  * k_batch_scan_convert: one block per matrix.  Warps stride over rows and
//    lanes over 16-byte vectors of a row (consecutive addresses); the block
//    folds the largest i-j / j-i over nonzeros, applies the dispatch predicate
//    and, for a banded matrix, writes its band storage (reading the band back
//    from the matrix it has just scanned, which is still in L2).
//  * k_batch_factor: one warp per pair of matrices, in place on their band
//    storage, in the xGBTRF order of operations.  Bands whose active window
//    fits a warp's lanes are factored with the window in registers
//    (window_gbtrf): no shared memory, one argmax, a few shuffles, one DMUL
//    and one DFMA per column, two matrices per warp instruction when both
//    windows fit 16 lanes; wider bands column by column (warp_gbtrf).
//  The band storage written by the first kernel (58.7 MB for 4096 matrices of
//  n = 256, kl = ku = 2) stays in L2 for the second.  (A single kernel with
//  scanner and factor warps side by side was slower: the factor warps' loads
//  queue behind the scanners' HBM stream.)
#include <climits>

#include "common.cuh"
#include "rcp.cuh"
#include "regwin.cuh"

namespace bandlu {
namespace {

__global__ void __launch_bounds__(256) k_batch_scan_convert(const double *__restrict__ A, long long n, long long lda,
                                                            long long strideA, long long batch, double *__restrict__ AB,
                                                            long long ldab, long long strideAB, int *__restrict__ d_kl,
                                                            int *__restrict__ d_ku, int *__restrict__ d_info,
                                                            int *__restrict__ d_status, int vec) {
  __shared__ int s_l[8], s_u[8];
  __shared__ int s_kl, s_ku, s_banded;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (long long b = blockIdx.x; b < batch; b += gridDim.x) {
    const double *Ab = A + b * strideA;
    int lmax = 0, umax = 0;
    if (vec) {
      const long long nv = (n + 1) / 2;
      for (long long i = warp; i < n; i += nw) {
        const ulonglong2 *row = reinterpret_cast<const ulonglong2 *>(Ab + i * lda);
        for (long long v0 = lane; v0 < nv; v0 += 32 * 4) {
          ulonglong2 x[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const long long v = v0 + 32 * u;
            x[u] = v < nv ? __ldcs(row + v) : make_ulonglong2(0ull, 0ull);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (((x[u].x << 1) | (x[u].y << 1)) != 0ull) {
              const long long j0 = 2 * (v0 + 32 * u);
              if (nz_bits(x[u].x)) {
                lmax = max(lmax, (int)(i - j0));
                umax = max(umax, (int)(j0 - i));
              }
              if (nz_bits(x[u].y) && j0 + 1 < n) {
                lmax = max(lmax, (int)(i - j0 - 1));
                umax = max(umax, (int)(j0 + 1 - i));
              }
            }
          }
        }
      }
    } else {
      for (long long i = warp; i < n; i += nw) {
        const unsigned long long *row = reinterpret_cast<const unsigned long long *>(Ab + i * lda);
        for (long long j = lane; j < n; j += 32) {
          if (nz_bits(__ldcs(row + j))) {
            lmax = max(lmax, (int)(i - j));
            umax = max(umax, (int)(j - i));
          }
        }
      }
    }
    lmax = __reduce_max_sync(FULL, lmax);
    umax = __reduce_max_sync(FULL, umax);
    if (lane == 0) {
      s_l[warp] = lmax;
      s_u[warp] = umax;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int kl = 0, ku = 0;
      for (int w = 0; w < nw; ++w) {
        kl = max(kl, s_l[w]);
        ku = max(ku, s_u[w]);
      }
      const bool banded = predicate_banded(n, kl, ku, ldab);
      s_kl = kl;
      s_ku = ku;
      s_banded = banded ? 1 : 0;
      d_kl[b] = kl;
      d_ku[b] = ku;
      d_info[b] = 0;
      d_status[b] = banded ? BANDLU_OK : BANDLU_NOT_BANDED;
    }
    __syncthreads();
    if (s_banded) {
      const long long kl = s_kl, ku = s_ku, kv = kl + ku;
      double *ABb = AB + b * strideAB;
      const long long total = n * ldab;
      for (long long e = threadIdx.x; e < total; e += blockDim.x) {
        const long long j = e / ldab;
        const long long r = e - j * ldab;
        const long long i = j - kv + r;
        double v = 0.0;
        if (r >= kl && r <= kv + kl && i >= 0 && i < n) v = Ab[i * lda + j];
        ABb[e] = v;
      }
    }
    __syncthreads();
  }
}

// Unblocked banded elimination by one warp on band storage `ab` (shared or
// global memory), in the xGBTRF order of operations.  32-bit indices (n < 2^31).
// Candidates of a pivot column sit one per lane; the first-max argmax is the
// exact integer reduction over |x|'s bit pattern.  Returns info.
__device__ int warp_gbtrf(double *ab, int ldab, int n, int kl, int ku, int *ipiv) {
  const int lane = threadIdx.x & 31;
  const int kv = kl + ku;
  if (kl > 0) {
    for (long long e = lane; e < (long long)n * kl; e += 32) {
      const long long c = e / kl, r = e - c * kl;
      ab[r + c * ldab] = 0.0;
    }
  }
  __syncwarp();
  int ju = 0;
  int info = 0;
  for (int j = 0; j < n; ++j) {
    const int km = min(kl, n - 1 - j);
    double *col = ab + (long long)j * ldab;
    int p;
    if (km < 32) {
      const double x = lane <= km ? col[kv + lane] : 0.0;
      bool allz;
      p = warp_argmax_first_z(lane <= km ? pivot_abs_key(x, lane == 0) : 0ull, &allz);
    } else {
      KeyIdx best{0ull, LLONG_MAX};
      for (int t = lane; t <= km; t += 32) best = better(best, KeyIdx{pivot_abs_key(col[kv + t], t == 0), t});
      p = (int)warp_reduce_keyidx(best).idx;
    }
    const double pv = col[kv + p];
    if (lane == 0) ipiv[j] = j + p + 1;
    if (nz(pv)) {
      ju = max(ju, min(j + ku + p, n - 1));
      if (p != 0) {
        for (int c = j + lane; c <= ju; c += 32) {
          double *x = ab + (kv + j - c) + (long long)c * ldab;
          double *y = ab + (kv + j + p - c) + (long long)c * ldab;
          const double t0 = *x;
          *x = *y;
          *y = t0;
        }
      }
      if (km > 0) {
        const double r = rcp_rn(pv);  // IEEE 1/pv on the integer pipes
        __syncwarp();
        for (int t = 1 + lane; t <= km; t += 32) col[kv + t] *= r;
        __syncwarp();
        const int ncol = ju - j;
        for (int e = lane; e < ncol * km; e += 32) {
          const int cc = e / km, t = 1 + (e - cc * km);
          const int c = j + 1 + cc;
          double *colc = ab + (long long)c * ldab;
          const double u = colc[kv + j - c];
          if (nz(u)) colc[kv + j + t - c] = fma(-col[kv + t], u, colc[kv + j + t - c]);
        }
      }
    } else if (info == 0) {
      info = j + 1;
    }
    __syncwarp();
  }
  return info;
}

// One warp per pair of matrices: both factored together in 16-lane windows
// when both bands fit one; otherwise one after the other (a 32-lane window,
// or column by column for wider bands).
__global__ void __launch_bounds__(128) k_batch_factor(long long n, long long batch, double *__restrict__ AB,
                                                      long long ldab, long long strideAB, int *__restrict__ ipiv,
                                                      long long strideP, const int *__restrict__ d_kl,
                                                      const int *__restrict__ d_ku, int *__restrict__ d_info,
                                                      const int *__restrict__ d_status, int win_ok) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, wpb = blockDim.x >> 5;
  const long long b0 = 2 * ((long long)blockIdx.x * wpb + warp);
  if (b0 >= batch) return;  // whole warp leaves together
  bool ok[2];
  int kl[2], ku[2];
  for (int t = 0; t < 2; ++t) {
    const long long b = b0 + t;
    ok[t] = b < batch && d_status[b] == BANDLU_OK;
    kl[t] = ok[t] ? d_kl[b] : 0;
    ku[t] = ok[t] ? d_ku[b] : 0;
  }
  auto fits = [&](int t, int width) { return win_ok && (kl[t] + 1) * (kl[t] + ku[t] + 1) <= width; };
  if (ok[0] && ok[1] && fits(0, 16) && fits(1, 16)) {
    double *const abp[2] = {AB + b0 * strideAB, AB + (b0 + 1) * strideAB};
    int *const pvp[2] = {ipiv + b0 * strideP, ipiv + (b0 + 1) * strideP};
    int info[2];
    regwin::window_gbtrf<2>(abp, (int)ldab, (int)n, kl, ku, pvp, info);
    if (lane == 0) {
      d_info[b0] = info[0];
      d_info[b0 + 1] = info[1];
    }
    return;
  }
  for (int t = 0; t < 2; ++t) {
    if (!ok[t]) continue;
    const long long b = b0 + t;
    double *ABb = AB + b * strideAB;
    int info;
    if (fits(t, 32)) {
      double *const abp[1] = {ABb};
      int *const pvp[1] = {ipiv + b * strideP};
      const int klt[1] = {kl[t]}, kut[1] = {ku[t]};
      int inf[1];
      regwin::window_gbtrf<1>(abp, (int)ldab, (int)n, klt, kut, pvp, inf);
      info = inf[0];
    } else {
      info = warp_gbtrf(ABb, (int)ldab, (int)n, kl[t], ku[t], ipiv + b * strideP);
    }
    if (lane == 0) d_info[b] = info;
  }
}


}  // namespace

int launch_batched(const double *A, int64_t n, int64_t lda, int64_t strideA, int64_t batch, double *AB, int64_t ldab,
                   int64_t strideAB, int *ipiv, int64_t strideP, int *d_kl, int *d_ku, int *d_info, int *d_status,
                   cudaStream_t s) {
  if (batch == 0) return BANDLU_OK;
  const int vec = ((reinterpret_cast<uintptr_t>(A) & 15u) == 0) && (lda % 2 == 0) && (strideA % 2 == 0);
  long long grid1 = batch;
  const long long cap = (long long)device_sms() * 64;
  if (grid1 > cap) grid1 = cap;
  k_batch_scan_convert<<<(unsigned)grid1, 256, 0, s>>>(A, n, lda, strideA, batch, AB, ldab, strideAB, d_kl, d_ku,
                                                       d_info, d_status, vec);
  BANDLU_CHECK_LAUNCH();
  if (n == 0) return BANDLU_OK;
  const int wpb = 4;
  const long long grid2 = ((batch + 1) / 2 + wpb - 1) / wpb;  // a warp per pair of matrices
  const int win_ok = (n + 1) * ldab < (int64_t)INT_MAX;  // 32-bit offsets in window_gbtrf
  k_batch_factor<<<(unsigned)grid2, 32 * wpb, 0, s>>>(n, batch, AB, ldab, strideAB, ipiv, strideP, d_kl, d_ku,
                                                      d_info, d_status, win_ok);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu
