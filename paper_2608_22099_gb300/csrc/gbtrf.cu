// gbtrf.cu -- banded LU with partial pivoting (Sec. II-A step 3; f(N) ~ O(N*P*Q), Eq. S-N-N3).
//
// Two single-matrix kernels:
//
//  * k_gbtrf_window (kl <= 27, the narrow bands the method targets).  One CTA.
//    The active part of the band at step j is the dense (kl+1) x (kv+1) block
//    of rows j..j+kl and columns j..j+kv.  It lives in shared memory in NATURAL
//    coordinates: R = kl+1+kDelta row slots (a ring of the active rows plus
//    rows prefetched kDelta steps ahead) times CS = kl+kv+1 column slots
//    (column c -> slot c mod CS).  A row interchange swaps two entries of the
//    logical-row -> slot map instead of moving data.  Warp 0 (the panel warp)
//    owns the critical path: it keeps the pivot column in registers (lane t =
//    row j+t), finds the pivot with an exact integer argmax, forms the
//    multipliers, and itself applies step j to column j+1 so that step j+1
//    can start at once.  Warps 1..3 (updaters) apply step j to columns
//    j+2..j+kv (column j+2 first, which the panel needs next), stream the
//    finished U row to global memory and prefetch the rows that enter the
//    window.  Hand-offs use mbarriers with bounded waits:
//      full[b]   panel -> updaters: step j's multipliers, row slots, zero-pivot flag
//      empty[b]  updaters -> panel and updaters: all updater warps finished step j
//      colready  warp 1 -> panel: column j+2 holds step j (and column j+1+kv is cleared)
//
//  * k_gbtrf_generic (any kl, ku).  One CTA works directly on AB in global
//    memory (the active window stays L2-resident), one column at a time.
//
// Both follow the xGBTRF order of operations exactly (first-max pivot,
// interchange, reciprocal then multiply, fma(-l, u, a) updates applied in
// column order, zero-u skip), so they reproduce the unblocked elimination
// bit for bit.  Entries of U beyond the running column reach ju are structural
// zeros in both interchanged rows, so interchanging and (skipped) updating the
// whole window is the same as LAPACK's restriction to columns j..ju.
#include <climits>

#include "common.cuh"
#include "sync.cuh"

namespace bandlu {
namespace {

constexpr int kDelta = 4;          // rows prefetched ahead of the active window
constexpr int kWinMaxKl = 31 - kDelta;
constexpr int kNU = 3;             // updater warps
constexpr int kNUT = 32 * kNU;     // updater threads

struct WinShared {
  unsigned long long full[2];   // panel -> updaters: step buffer b is published
  unsigned long long empty[2];  // updaters -> panel: step buffer b is consumed
  unsigned long long colready;  // warp 1 -> panel: column j+2 holds step j
  int abort_flag;
  int zp[2];
  int slot[2][32];
  double l[2][32];
};

template <int PF>
__global__ void __launch_bounds__(128, 1) k_gbtrf_window(long long n, int kl, int ku, double *__restrict__ AB,
                                                          long long ldab, int *__restrict__ ipiv,
                                                          int *__restrict__ d_info) {
  extern __shared__ double W[];  // R * CS
  __shared__ WinShared sh;
  const int kv = kl + ku;
  const int R = kl + 1 + kDelta;
  const int CS = kl + kv + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&sh.full[0], 1);
    mbar_init(&sh.full[1], 1);
    mbar_init(&sh.empty[0], kNU);
    mbar_init(&sh.empty[1], kNU);
    mbar_init(&sh.colready, 1);
    sh.abort_flag = 0;
  }
  // Fill-row entries of the top-left corner (element row < 0) are cleared, as
  // the elimination clears every fill row before it starts.
  for (int e = threadIdx.x; e < kl * kv; e += blockDim.x) {
    const int r = e / kv, c = e - r * kv;
    if (c < kv - r && c < n) AB[r + (long long)c * ldab] = 0.0;
  }
  // Rows 0..R-1 go to slots 0..R-1; row i covers columns i-kl .. i+kv.
  const int R0 = (int)min((long long)R, n);
  for (int e = threadIdx.x; e < R0 * CS; e += blockDim.x) {
    const int i = e / CS, k = e - i * CS;
    const long long c = (long long)i - kl + k;
    double v = 0.0;
    if (c >= 0 && c < n && c <= i + ku) v = AB[(kv + i - c) + c * ldab];
    const int q = (int)(((c % CS) + CS) % CS);
    W[i * CS + q] = v;
  }
  __syncthreads();

  int info = 0;
  if (warp == 0) {
    // ---------------- panel warp ----------------
    int slot_reg = lane;  // slot of logical row j+lane (lanes < R)
    double cur = (lane <= kl && lane < n) ? W[lane * CS] : 0.0;
    int qn = 1 % CS;  // column slot of column j+1
    for (long long j = 0; j < n; ++j) {
      const int km = (int)min((long long)kl, n - 1 - j);
      const bool valid = lane <= km;
      const unsigned long long key = valid ? abs_key(cur) : 0ull;
      // Every candidate's reciprocal is formed while the argmax runs.
      const double rl = 1.0 / ((valid && nz(cur)) ? cur : 1.0);
      const int p = warp_argmax_first(key);
      const double pv = __shfl_sync(FULL, cur, p);
      const double r = __shfl_sync(FULL, rl, p);
      const double c0 = __shfl_sync(FULL, cur, 0);
      const bool zp = !nz(pv);  // exact zero pivot (then p == 0)
      if (lane == p) cur = c0;
      if (lane == 0) cur = pv;
      const int s0 = __shfl_sync(FULL, slot_reg, 0);
      const int sp = __shfl_sync(FULL, slot_reg, p);
      if (lane == p) slot_reg = s0;
      if (lane == 0) slot_reg = sp;
      const double l = (!zp && lane >= 1 && valid) ? cur * r : cur;
      if (lane == 0) {
        ipiv[j] = (int)(j + p + 1);
        AB[kv + j * ldab] = pv;
      }
      if (lane >= 1 && valid) AB[(kv + lane) + j * ldab] = l;
      if (zp && info == 0) info = (int)(j + 1);
      const int b = (int)(j & 1);
      if (j >= 1 && !mbar_wait_warp(&sh.colready, (unsigned)((j - 1) & 1), &sh.abort_flag)) break;
      if (j >= 2 && !mbar_wait_warp(&sh.empty[b], (unsigned)(((j - 2) >> 1) & 1), &sh.abort_flag)) break;
      sh.l[b][lane] = l;
      sh.slot[b][lane] = slot_reg;
      if (lane == 0) sh.zp[b] = zp ? 1 : 0;
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.full[b]);
      if (j + 1 < n) {
        // column j+1, logical rows j .. j+kl+1 (holds steps <= j-1)
        double v = 0.0;
        if (lane <= kl + 1 && j + lane < n) v = W[slot_reg * CS + qn];
        // U(j, j+1); when kv == 0 (diagonal matrix) column j+1 lies outside row j's band
        const double u = kv >= 1 ? __shfl_sync(FULL, v, 0) : 0.0;
        if (lane == 0 && kv >= 1) AB[(kv - 1) + (j + 1) * ldab] = u;
        if (!zp && nz(u) && lane >= 1 && valid) v = fma(-l, u, v);
        cur = __shfl_down_sync(FULL, v, 1);  // logical rows j+1 .. j+1+kl
      }
      const int sfirst = __shfl_sync(FULL, slot_reg, 0);
      const int sn = __shfl_down_sync(FULL, slot_reg, 1);
      slot_reg = (lane == R - 1) ? sfirst : sn;  // retired row's slot takes row j+R
      qn = (qn + 1 == CS) ? 0 : qn + 1;
    }
  } else if (warp <= kNU) {
    // ---------------- updater warps ----------------
    const int tid_u = threadIdx.x - 32;
    double pf[PF];
    bool have_pf = false;
    long long pf_row = 0;
    int pf_slot = 0;
    int qj = 0;  // column slot of column j
    for (long long j = 0; j < n; ++j) {
      const int b = (int)(j & 1);
      if (!mbar_wait_warp(&sh.full[b], (unsigned)((j >> 1) & 1), &sh.abort_flag)) break;
      // Consecutive steps update the same entries through different threads: every
      // updater warp must have finished step j-1 before any starts step j.
      if (j >= 1 && !mbar_wait_warp(&sh.empty[b ^ 1], (unsigned)(((j - 1) >> 1) & 1), &sh.abort_flag)) break;
      const int km = (int)min((long long)kl, n - 1 - j);
      const bool zp = sh.zp[b] != 0;
      const long long cmax = min(j + kv, n - 1);
      const int s0 = sh.slot[b][0];
      if (warp == 1) {
        const long long c = j + 2;
        if (c <= cmax) {
          int q = qj + 2;
          if (q >= CS) q -= CS;
          const double u = W[s0 * CS + q];
          if (lane == 0) AB[(kv - 2) + c * ldab] = u;
          if (!zp && nz(u) && lane >= 1 && lane <= km) {
            const int st = sh.slot[b][lane];
            W[st * CS + q] = fma(-sh.l[b][lane], u, W[st * CS + q]);
          }
        }
        // Column j+1+kv enters the window at step j+1.  Rows j+1..j+kl (any
        // physical row pushed down by interchanges) hold structural zeros there;
        // their slots may still hold a column that left the window CS steps ago.
        if (lane >= 1 && lane <= kl && j + 1 + kv < n) {
          int qe = qj + 1 + kv;
          if (qe >= CS) qe -= CS;
          W[sh.slot[b][lane] * CS + qe] = 0.0;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.colready);
      }
      const long long ncols = cmax - (j + 2);
      if (ncols > 0) {
        const int rows = km + 1;
        const int tot = (int)ncols * rows;
        for (int e = tid_u; e < tot; e += kNUT) {
          const int cc = e / rows, t = e - cc * rows;
          const long long c = j + 3 + cc;
          int q = qj + 3 + cc;
          if (q >= CS) q -= CS;
          const double u = W[s0 * CS + q];
          if (t == 0) {
            AB[(kv + j - c) + c * ldab] = u;  // U(j, c)
          } else if (!zp && nz(u)) {
            const int st = sh.slot[b][t];
            W[st * CS + q] = fma(-sh.l[b][t], u, W[st * CS + q]);
          }
        }
      }
      // The row fetched one step ago goes into its slot (the slot's previous
      // row retired two steps ago).
      if (have_pf) {
#pragma unroll
        for (int k = 0; k < PF; ++k) {
          const int kk = tid_u + k * kNUT;
          if (kk < CS) W[pf_slot * CS + (int)((pf_row - kl + kk) % CS)] = pf[k];
        }
        have_pf = false;
      }
      // Fetch row j-1+R: its band entries, zeros for the rest of its columns.
      if (j >= 1 && j - 1 + R < n) {
        const long long i = j - 1 + R;
        pf_row = i;
        pf_slot = sh.slot[b][R - 1];
        have_pf = true;
#pragma unroll
        for (int k = 0; k < PF; ++k) {
          const int kk = tid_u + k * kNUT;
          const long long c = i - kl + kk;
          pf[k] = (kk < CS && c <= i + ku && c < n) ? AB[(kv + i - c) + c * ldab] : 0.0;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.empty[b]);
      qj = (qj + 1 == CS) ? 0 : qj + 1;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *d_info = sh.abort_flag ? -BANDLU_ERR_TIMEOUT : info;
}

__global__ void __launch_bounds__(1024) k_gbtrf_generic(long long n, int kl, int ku, double *__restrict__ AB,
                                                         long long ldab, int *__restrict__ ipiv,
                                                         int *__restrict__ d_info) {
  __shared__ KeyIdx s_red[32];
  __shared__ int s_p;
  __shared__ double s_r;
  const long long kv = (long long)kl + ku;
  const int tid = threadIdx.x, B = blockDim.x, lane = tid & 31, warp = tid >> 5, nw = B >> 5;
  if (kl > 0) {
    for (long long e = tid; e < n * kl; e += B) {
      const long long c = e / kl, r = e - c * kl;
      AB[r + c * ldab] = 0.0;
    }
  }
  __syncthreads();
  long long ju = 0;
  int info = 0;
  for (long long j = 0; j < n; ++j) {
    const long long km = min((long long)kl, n - 1 - j);
    double *colj = AB + j * ldab;
    KeyIdx best{0ull, LLONG_MAX};
    for (long long t = tid; t <= km; t += B) best = better(best, KeyIdx{abs_key(colj[kv + t]), t});
    best = warp_reduce_keyidx(best);
    if (lane == 0) s_red[warp] = best;
    __syncthreads();
    if (warp == 0) {
      KeyIdx v = lane < nw ? s_red[lane] : KeyIdx{0ull, LLONG_MAX};
      v = warp_reduce_keyidx(v);
      if (lane == 0) s_p = (int)v.idx;
    }
    __syncthreads();
    const long long p = s_p;
    const double piv = colj[kv + p];
    if (tid == 0) ipiv[j] = (int)(j + p + 1);
    if (nz(piv)) {
      ju = max(ju, min(j + ku + p, n - 1));
      if (p != 0) {
        for (long long c = j + tid; c <= ju; c += B) {
          double *x = AB + (kv + j - c) + c * ldab;
          double *y = AB + (kv + j + p - c) + c * ldab;
          const double t0 = *x;
          *x = *y;
          *y = t0;
        }
        __syncthreads();
      }
      if (km > 0) {
        if (tid == 0) s_r = 1.0 / colj[kv];
        __syncthreads();
        const double r = s_r;
        for (long long t = 1 + tid; t <= km; t += B) colj[kv + t] *= r;
        __syncthreads();
        const long long tot = (ju - j) * km;
        for (long long e = tid; e < tot; e += B) {
          const long long cc = e / km, t = 1 + (e - cc * km);
          const long long c = j + 1 + cc;
          double *colc = AB + c * ldab;
          const double u = colc[kv + j - c];
          if (nz(u)) colc[kv + j + t - c] = fma(-colj[kv + t], u, colc[kv + j + t - c]);
        }
        __syncthreads();
      }
    } else if (info == 0) {
      info = (int)(j + 1);
    }
  }
  if (tid == 0) *d_info = info;
}

template <int PF>
int launch_window(long long n, int kl, int ku, double *AB, long long ldab, int *ipiv, int *d_info, size_t smem,
                  cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(k_gbtrf_window<PF>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024) !=
        cudaSuccess)
      return BANDLU_ERR_CUDA;
    attr = true;
  }
  k_gbtrf_window<PF><<<1, 128, smem, s>>>(n, kl, ku, AB, ldab, ipiv, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace

int launch_gbtrf(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t s) {
  if (n == 0) {
    if (cudaMemsetAsync(d_info, 0, sizeof(int), s) != cudaSuccess) return BANDLU_ERR_CUDA;
    return BANDLU_OK;
  }
  const long long kv = (long long)kl + ku;
  const long long CS = kl + kv + 1;
  const long long R = kl + 1 + kDelta;
  const size_t smem = (size_t)(R * CS) * sizeof(double);
  if (kl <= kWinMaxKl && CS <= 8 * kNUT && smem <= 200 * 1024) {
    const int pf = (int)((CS + kNUT - 1) / kNUT);
    if (pf <= 1) return launch_window<1>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
    if (pf <= 2) return launch_window<2>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
    if (pf <= 4) return launch_window<4>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
    return launch_window<8>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
  }
  k_gbtrf_generic<<<1, 1024, 0, s>>>(n, kl, ku, AB, ldab, ipiv, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu
