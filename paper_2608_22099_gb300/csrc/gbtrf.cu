// gbtrf.cu -- banded LU with partial pivoting (Sec. II-A step 3; f(N) ~ O(N*P*Q), Eq. S-N-N3).
//
// Two single-matrix kernels here, after the narrowest bands (a one-warp
// register window, k_gbtrf_regwin) and before the wide ones (the multi-CTA
// kernel of gbtrf_wide.cu, when it can be launched):
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
//    can start at once.  The helper warp applies step j to column j+2 (which
//    the panel needs next), 11 updater warps (none on the panel's SMSP) to
//    columns j+3..j+kv and write the finished U row, and the I/O warp writes
//    the pivot and multipliers and copies the rows that enter the window into
//    their slots (cp.async).  Hand-offs are two named barriers per step (see
//    kBarPub/kBarCol).  (Two more updater warps on the panel's SMSP were
//    measured: faster for kl = 27, slower for kl <= 16, where the panel's
//    FP64 instructions then queue behind theirs.)
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
#include "rcp.cuh"
#include "regwin.cuh"
#include "sync.cuh"

namespace bandlu {
namespace {

constexpr int kDelta = 4;          // rows prefetched ahead of the active window
constexpr int kWinMaxKl = 31 - kDelta;
constexpr int kWarps = 16;         // warp 0 panel, 4 helper, 13 I/O, 11 updaters, 8 and 12 idle
constexpr int kNU = 11;            // updater warps: every warp w with w % 4 != 0 except kIoWarp
constexpr int kNUT = 32 * kNU;     // updater threads
constexpr int kHelperWarp = 4;     // shares the panel's SMSP (shared-memory work only)
constexpr int kIoWarp = 13;        // global stores and row prefetch, away from the panel's SMSP

// One published row of step j: its multiplier (the pivot itself for row 0) and
// the offset of its slot in W.
struct __align__(16) RowPk {
  double l;
  int rb;   // slot * CS
  int pad;
};

struct __align__(16) StepMeta {
  double u1;  // U(j, j+1)
  int zp;     // exact zero pivot
  int p;      // pivot offset
};


// Named barriers of the window kernel (0 is __syncthreads):
//   kBarPub: the panel arrives once step j (multipliers, row slots, pivot) is
//            published; the 12 updater warps and the helper warp sync on it, so
//            it also orders all their step j-1 work before any step j.
//   kBarCol: the helper warp arrives once column j+2 holds step j (and column
//            j+1+kv is cleared); the panel syncs on it before it reads column j+2.
// Every participating warp runs exactly n steps and executes its barrier
// operations unconditionally, once per step.  The panel arrives at kBarPub(j)
// only after kBarCol(j-1), which the helper reaches only after kBarPub(j-1)
// completed, and the helper arrives at kBarCol(j) only after kBarPub(j)
// completed, which needs the panel's arrival after kBarCol(j-1): the phases of
// both barriers alternate.
constexpr int kBarPub = 1, kBarCol = 2;
constexpr int kPubCount = 32 * (1 + kNU + 2);

#ifdef BANDLU_BOUNDED_SYNC
// Checked build (development and tests only): the same protocol on mbarriers
// with bounded waits.  A protocol slip (a missing participant, a miscounted
// barrier) ends the kernel with info = -BANDLU_ERR_TIMEOUT instead of a hang.
struct BarState {
  unsigned long long mb[3];
  int abort_flag;
};
__device__ __forceinline__ void bar_init(BarState &st) {
  mbar_init(&st.mb[kBarPub], kPubCount / 32);
  mbar_init(&st.mb[kBarCol], 2);
  st.abort_flag = 0;
}
__device__ __forceinline__ void bar_arrive_x(BarState &st, int id) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&st.mb[id]);
}
// phase: how many times this warp has synced on barrier `id` so far
__device__ __forceinline__ bool bar_sync_x(BarState &st, int id, unsigned &phase) {
  bar_arrive_x(st, id);
  const bool ok = mbar_wait_warp(&st.mb[id], phase & 1u, &st.abort_flag);
  ++phase;
  return ok;
}
#define BAR_SYNC(id, count, phase) bar_sync_x(sh.bars, (id), (phase))
#define BAR_ARRIVE(id, count) bar_arrive_x(sh.bars, (id))
#define BAR_FAILED() (sh.bars.abort_flag != 0)
#else
__device__ __forceinline__ bool bar_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
  return true;
}
__device__ __forceinline__ void bar_arrive(int id, int count) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}
#define BAR_SYNC(id, count, phase) bar_sync((id), (count))
#define BAR_ARRIVE(id, count) bar_arrive((id), (count))
#define BAR_FAILED() false
#endif

struct WinShared {
  StepMeta meta[2];
  double u2[2];  // U(j, j+2), from the helper to the I/O warp
  RowPk pk[2][32];
#ifdef BANDLU_BOUNDED_SYNC
  BarState bars;
#endif
};


// Asynchronous global -> shared copies (the I/O warp's row prefetch).
__device__ __forceinline__ void cp_async8(double *dst, const double *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"((unsigned)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
// every group but the newest has completed
__device__ __forceinline__ void cp_async_wait_prior() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Out of line, so that the rarely taken division is not if-converted into the
// pivot chain of the panel warp.
__device__ __noinline__ double div_slow(double x) { return 1.0 / x; }

// The window factorisation (kWarps warps; W: R * CS doubles of dynamic shared
// memory), for k_gbtrf_window and the device-side dispatch.
template <int K, int PF>
__device__ __forceinline__ void window_factor(int n, int kl, int ku, double *__restrict__ AB, long long ldab,
                                              int *__restrict__ ipiv, int *__restrict__ d_info, double *W,
                                              WinShared &sh) {
  const int kv = kl + ku;
  const int R = kl + 1 + kDelta;
  const int CS = kl + kv + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

#ifdef BANDLU_BOUNDED_SYNC
  if (threadIdx.x == 0) bar_init(sh.bars);
#endif
  // Fill-row entries of the top-left corner (element row < 0) are cleared, as
  // the elimination clears every fill row before it starts.
  for (int e = threadIdx.x; e < kl * kv; e += blockDim.x) {
    const int r = e / kv, c = e - r * kv;
    if (c < kv - r && c < n) AB[r + (long long)c * ldab] = 0.0;
  }
  // Rows 0..R-1 go to slots 0..R-1; row i covers columns i-kl .. i+kv.
  const int R0 = min(R, n);
  for (int e = threadIdx.x; e < R0 * CS; e += blockDim.x) {
    const int i = e / CS, k = e - i * CS;
    const int c = i - kl + k;
    double v = 0.0;
    if (c >= 0 && c < n && c <= i + ku) v = AB[(kv + i - c) + (long long)c * ldab];
    const int q = ((c % CS) + CS) % CS;
    W[i * CS + q] = v;
  }
  __syncthreads();

  int info = 0;
  if (warp == 0) {
    // ---------------- panel warp: the pivot chain only ----------------
    int slot_reg = lane;  // slot of logical row j+lane (lanes < R)
    double cur = (lane <= kl && lane < n) ? W[lane * CS] : 0.0;
    int qn = 1 % CS;  // column slot of column j+1
    unsigned ph_col = 0;
    for (int j = 0; j < n; ++j) {
      const int km = min(kl, n - 1 - j);
      const bool valid = lane <= km;
      // every lane forms the reciprocal of its own candidate while the argmax
      // runs; the pivot's is then taken from the winning lane
      bool myspec;
      const double myr = rcp_rn_fast(cur, &myspec);  // integer pipes
      bool zp;  // exact zero pivot (then p == 0)
      // (the two-pass form: here the shortcut's branch costs the panel more than
      // the second reduction it saves)
      const int p = regwin::argmax_two_pass(valid ? pivot_abs_key(cur, lane == 0) : 0ull, &zp);
      // interchange rows j and j+p: lanes 0 and p trade their values and slots
      const int src = lane == 0 ? p : (lane == p ? 0 : lane);
      slot_reg = __shfl_sync(FULL, slot_reg, src);
      // column j+1, logical rows j .. j+kl+1 (holds steps <= j-1): the load is
      // issued here and lands while the reciprocal is formed
      if (j >= 1 && !BAR_SYNC(kBarCol, 64, ph_col)) break;
      double v = 0.0;
      if (j + 1 < n && lane <= kl + 1 && j + lane < n) v = W[slot_reg * CS + qn];
      double r = __shfl_sync(FULL, myr, p);
      const bool rspec = __shfl_sync(FULL, myspec ? 1 : 0, p) != 0;
      if (rspec && !zp) r = div_slow(__shfl_sync(FULL, cur, p));  // subnormal / huge pivot: plain division
      cur = __shfl_sync(FULL, cur, src);
      // U(j, j+1); when kv == 0 (diagonal matrix) column j+1 lies outside row j's band
      const double u = kv >= 1 ? __shfl_sync(FULL, v, 0) : 0.0;
      const double l = (!zp && lane >= 1 && valid) ? cur * r : cur;
      // step j on column j+1 before the updaters' multiply-adds start competing
      // for the FP64 unit
      if (j + 1 < n && !zp && nz(u) && lane >= 1 && valid) v = fma(-l, u, v);
      // buffer b was last read in step j-2, which every reader finished before
      // the helper reached kBarCol(j-1)
      const int b = j & 1;
      sh.pk[b][lane].l = l;
      sh.pk[b][lane].rb = slot_reg * CS;
      if (lane == 0) {
        sh.meta[b].u1 = u;
        sh.meta[b].zp = zp ? 1 : 0;
        sh.meta[b].p = p;
      }
      __syncwarp();
      BAR_ARRIVE(kBarPub, kPubCount);
      cur = __shfl_down_sync(FULL, v, 1);  // logical rows j+1 .. j+1+kl
      if (zp && info == 0) info = j + 1;
      // retired row j's slot takes row j+R
      slot_reg = __shfl_sync(FULL, slot_reg, lane == R - 1 ? 0 : lane + 1);
      qn = (qn + 1 == CS) ? 0 : qn + 1;
    }
    if (!BAR_FAILED()) BAR_SYNC(kBarCol, 64, ph_col);  // the helper's arrival of the last step
  } else if (warp == kHelperWarp) {
    // ---------------- helper warp: column j+2 and the hand-off ----------------
    int qj = 0;
    unsigned ph_pub = 0;
    for (int j = 0; j < n; ++j) {
      const int b = j & 1;
      if (!BAR_SYNC(kBarPub, kPubCount, ph_pub)) break;
      const int km = min(kl, n - 1 - j);
      const bool zp = sh.meta[b].zp != 0;
      const int rb0 = sh.pk[b][0].rb;
      if (j + 2 <= min(j + kv, n - 1)) {
        int q = qj + 2;
        if (q >= CS) q -= CS;
        const double u = W[rb0 + q];
        if (lane == 0) sh.u2[b] = u;  // U(j, j+2), written out by the I/O warp
        if (!zp && nz(u) && lane >= 1 && lane <= km) {
          const RowPk pk = sh.pk[b][lane];
          W[pk.rb + q] = fma(-pk.l, u, W[pk.rb + q]);
        }
      }
      // Column j+1+kv enters the window at step j+1.  Rows j+1..j+kl (any
      // physical row pushed down by interchanges) hold structural zeros there;
      // their slots may still hold a column that left the window CS steps ago.
      if (lane >= 1 && lane <= kl && j + 1 + kv < n) {
        int qe = qj + 1 + kv;
        if (qe >= CS) qe -= CS;
        W[sh.pk[b][lane].rb + qe] = 0.0;
      }
      __syncwarp();
      BAR_ARRIVE(kBarCol, 64);
      qj = (qj + 1 == CS) ? 0 : qj + 1;
    }
  } else if (warp == kIoWarp) {
    // ---------------- I/O warp ----------------
    // Step j's pivot, U diagonal, U(j, j+1), U(j, j+2) and multipliers go to
    // global memory; then the row prefetch: row j-1+R enters the slot that row
    // j-1 left, copied straight into it with cp.async.  The copy issued in step
    // j is waited for at the end of step j+1, before this warp's arrival at
    // kBarPub(j+2): the row is first read in step j+3 (the panel's column j+4,
    // after kBarCol(j+2), which the helper reaches after kBarPub(j+2)), and the
    // load has two steps to land instead of stalling every step on it.
    int pfo[PF];
#pragma unroll
    for (int k = 0; k < PF; ++k) pfo[k] = (kDelta + lane + 32 * k) % CS;
    int qj = 0;
    unsigned ph_pub = 0;
    for (int j = 0; j < n; ++j) {
      const int b = j & 1;
      if (!BAR_SYNC(kBarPub, kPubCount, ph_pub)) break;
      const int km = min(kl, n - 1 - j);
      // U(j, j+2) of the previous step: the helper wrote it before kBarPub(j)
      if (lane == 0 && j >= 1 && kv >= 2 && j + 1 < n) AB[(kv - 2) + (long long)(j + 1) * ldab] = sh.u2[b ^ 1];
      if (lane == 0) {
        ipiv[j] = j + sh.meta[b].p + 1;
        AB[kv + (long long)j * ldab] = sh.pk[b][0].l;
        if (kv >= 1 && j + 1 < n) AB[(kv - 1) + (long long)(j + 1) * ldab] = sh.meta[b].u1;
      }
      if (lane >= 1 && lane <= km) AB[(kv + lane) + (long long)j * ldab] = sh.pk[b][lane].l;
      if (j >= 1 && j - 1 + R < n) {
        const int i = j - 1 + R;
        const int rb = sh.pk[b][R - 1].rb;
#pragma unroll
        for (int k = 0; k < PF; ++k) {
          const int kk = lane + 32 * k;
          if (kk < CS) {
            int q = qj + pfo[k];
            if (q >= CS) q -= CS;
            const int c = i - kl + kk;  // >= 0
            if (c <= i + ku && c < n)
              cp_async8(W + rb + q, AB + (kv + i - c) + (long long)c * ldab);
            else
              W[rb + q] = 0.0;
          }
        }
      }
      cp_async_commit();
      cp_async_wait_prior();  // the copy of step j-1 has landed
      qj = (qj + 1 == CS) ? 0 : qj + 1;
    }
    cp_async_wait_all();
  } else if ((warp & 3) != 0) {
    // ---------------- updater warps: columns j+3 .. j+kv ----------------
    // Updater index of this warp.  The order puts the warps that also take the
    // last, partial round of elements on different SMSPs, so that the FP64
    // instructions of a step spread evenly over the SMSPs' pipes.
    // warp -> updater index {-, 0, 2, 3, -, 1, 4, 5, -, 6, 7, 8, -, -, 9, 10}, four bits
    // per warp in one constant (a table would be a local-memory array)
    constexpr unsigned long long kUwPacked = 0xA9FF876F541F320Full;
    const int uw = (int)((kUwPacked >> (4 * warp)) & 15ull);  // 0..kNU-1
    const int tid_u = uw * 32 + lane;
    const int ncols = kv > 2 ? kv - 2 : 0;
    const int E = ncols * (kl + 1);
    const int EF = ncols * kl;  // elements with a multiply-add (rows t >= 1)
    // Static element map, columns fastest: elements 0..EF-1 are row offsets
    // t = 1 + e / ncols, column offsets d = 3 + e % ncols; the last ncols
    // elements are the U row (t = 0), which is only written out.  The lanes of
    // a warp read one row record (a broadcast) and consecutive columns of the
    // pivot row and of their own row (no bank conflicts), and every warp
    // instruction of the multiply-adds is full except the last.
    int ed[K], et[K];
    long long uoff[K];  // offset of U(j, j+d) in AB relative to column j
#pragma unroll
    for (int k = 0; k < K; ++k) {
      const int e = tid_u + kNUT * k;
      if (e < EF) {
        et[k] = 1 + e / ncols;
        ed[k] = 3 + (e - (et[k] - 1) * ncols);
      } else if (e < E) {
        et[k] = 0;
        ed[k] = 3 + (e - EF);
      } else {
        et[k] = 0;
        ed[k] = 0;
      }
      uoff[k] = (kv - ed[k]) + (long long)ed[k] * ldab;
    }
    int qj = 0;  // column slot of column j
    unsigned ph_pub = 0;
    for (int j = 0; j < n; ++j) {
      const int b = j & 1;
      if (!BAR_SYNC(kBarPub, kPubCount, ph_pub)) break;
      const int km = min(kl, n - 1 - j);
      const bool zp = sh.meta[b].zp != 0;
      const int cmax = min(j + kv, n - 1);
      const int rb0 = sh.pk[b][0].rb;
      // all loads first, then the fused multiply-adds, then the stores
      const bool full = j + kv <= n - 1;  // every mapped element is inside the matrix
      double *ABj = AB + (long long)j * ldab;
      double uu[K], xx[K], ll[K];
      int rr[K], qq[K];
      bool act[K];
#pragma unroll
      for (int k = 0; k < K; ++k) {
        act[k] = ed[k] != 0 && (full || (j + ed[k] <= cmax && et[k] <= km));
        int q = qj + ed[k];
        if (q >= CS) q -= CS;
        qq[k] = q;
        uu[k] = act[k] ? W[rb0 + q] : 0.0;
        const RowPk pk = sh.pk[b][et[k]];
        ll[k] = pk.l;
        rr[k] = pk.rb;
      }
#pragma unroll
      for (int k = 0; k < K; ++k) xx[k] = (act[k] && et[k] > 0) ? W[rr[k] + qq[k]] : 0.0;
#pragma unroll
      for (int k = 0; k < K; ++k) {
        if (!act[k]) continue;
        if (et[k] == 0) {
          ABj[uoff[k]] = uu[k];  // U(j, j+d)
        } else if (!zp && nz(uu[k])) {
          W[rr[k] + qq[k]] = fma(-ll[k], uu[k], xx[k]);
        }
      }
      qj = (qj + 1 == CS) ? 0 : qj + 1;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *d_info = BAR_FAILED() ? -BANDLU_ERR_TIMEOUT : info;
}

template <int K, int PF>
__global__ void __launch_bounds__(kWarps * 32, 1) k_gbtrf_window(int n, int kl, int ku, double *__restrict__ AB,
                                                                  long long ldab, int *__restrict__ ipiv,
                                                                  int *__restrict__ d_info) {
  extern __shared__ double W[];  // R * CS
  __shared__ WinShared sh;
  window_factor<K, PF>(n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
}

// Column-by-column elimination by the whole block (any block size) on AB in
// global memory, for k_gbtrf_generic and the device-side dispatch.
__device__ __forceinline__ void generic_factor(long long n, int kl, int ku, double *__restrict__ AB, long long ldab,
                                               int *__restrict__ ipiv, int *__restrict__ d_info) {
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
    for (long long t = tid; t <= km; t += B) best = better(best, KeyIdx{pivot_abs_key(colj[kv + t], t == 0), t});
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

__global__ void __launch_bounds__(1024) k_gbtrf_generic(long long n, int kl, int ku, double *__restrict__ AB,
                                                         long long ldab, int *__restrict__ ipiv,
                                                         int *__restrict__ d_info) {
  generic_factor(n, kl, ku, AB, ldab, ipiv, d_info);
}

// The narrowest bands, (kl+1)*(kl+ku+1) <= 32: one warp with the active window
// in registers (regwin.cuh).  Fill-row entries above the matrix are cleared
// first, as the elimination clears every fill row; the window writes the rest.
// Called by one whole warp.
__device__ __forceinline__ void regwin_factor(int n, int kl, int ku, double *__restrict__ AB, int ldab,
                                              int *__restrict__ ipiv, int *__restrict__ d_info) {
  const int kv = kl + ku, lane = threadIdx.x & 31;
  if (kl > 0) {
    for (int e = lane; e < kl * min(n, kv); e += 32) {
      const int jj = e / kl, rr = e - jj * kl;
      if (rr < kv - jj) AB[rr + jj * ldab] = 0.0;
    }
  }
  __syncwarp();
  double *const abp[1] = {AB};
  int *const pvp[1] = {ipiv};
  const int klv[1] = {kl}, kuv[1] = {ku};
  int info[1];
  regwin::window_gbtrf<1>(abp, ldab, n, klv, kuv, pvp, info);
  if (lane == 0) *d_info = info[0];
}

__global__ void __launch_bounds__(32) k_gbtrf_regwin(int n, int kl, int ku, double *__restrict__ AB, int ldab,
                                                     int *__restrict__ ipiv, int *__restrict__ d_info) {
  regwin_factor(n, kl, ku, AB, ldab, ipiv, d_info);
}

// The path choice of launch_gbtrf (without the multi-CTA kernel), shared by the
// host launcher and the device-side dispatch: 0 register window, 1 shared-
// memory window (*K, *PF: its template parameters, *smem: its bytes), 2 generic.
__host__ __device__ inline int factor_path(long long n, int kl, int ku, long long ldab, int *K, int *PF,
                                           size_t *smem) {
  const long long kv = (long long)kl + ku;
  if ((kl + 1LL) * (kv + 1) <= 32 && (n + 1) * ldab < (long long)INT_MAX) return 0;
  const long long CS = kl + kv + 1;
  const long long R = kl + 1 + kDelta;
  *smem = (size_t)(R * CS) * sizeof(double);
  const long long E = kv > 2 ? (kv - 2) * (kl + 1) : 0;  // trailing elements per step
  if (kl <= kWinMaxKl && CS <= 8 * 32 && E <= 8 * kNUT && *smem <= 200 * 1024) {
    const int pf = (int)((CS + 31) / 32);
    const int k = (int)((E + kNUT - 1) / kNUT);
    *PF = pf <= 1 ? 1 : (pf <= 2 ? 2 : (pf <= 4 ? 4 : 8));
    *K = k <= 1 ? 1 : (k <= 2 ? 2 : (k <= 4 ? 4 : 8));
    return 1;
  }
  return 2;
}

template <int K>
__device__ __forceinline__ void window_factor_pf(int PF, int n, int kl, int ku, double *AB, long long ldab, int *ipiv,
                                                 int *d_info, double *W, WinShared &sh) {
  if (PF == 1) window_factor<K, 1>(n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
  else if (PF == 2) window_factor<K, 2>(n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
  else if (PF == 4) window_factor<K, 4>(n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
  else window_factor<K, 8>(n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
}

// Device-side dispatch: the factorisation of dispatch_lu_async, with (kl, ku)
// and the dispatch decision read from device memory.  kWarps warps and
// smem_bytes of dynamic shared memory, enough for every shared-memory window
// that fits the band storage (2*kl+ku+1 <= ldab); the block takes the path
// launch_gbtrf would take, except that bands beyond the windows run the
// block-wide generic elimination (the multi-CTA kernel's grid and scratch are
// sized from kl on the host).
__global__ void __launch_bounds__(kWarps * 32, 1) k_gbtrf_on_device(int n, double *__restrict__ AB, long long ldab,
                                                                     int *__restrict__ ipiv,
                                                                     const int *__restrict__ d_kl,
                                                                     const int *__restrict__ d_ku,
                                                                     const int *__restrict__ d_status,
                                                                     int *__restrict__ d_info, size_t smem_bytes,
                                                                     int wide_rows_cap, int *__restrict__ wide_flag) {
  extern __shared__ double W[];
  __shared__ WinShared sh;
  if (*d_status != BANDLU_OK) return;  // declined: nothing is written
  const int kl = *d_kl, ku = *d_ku;
  int K = 1, PF = 1;
  size_t smem = 0;
  int path = factor_path(n, kl, ku, ldab, &K, &PF, &smem);
  if (path == 1 && smem > smem_bytes) path = 2;
  if (path == 2 && wide_flag != nullptr && wide_pair_takes(n, kl, ku, wide_rows_cap)) {
    // the cluster-pair kernel enqueued after this one factors the band
    if (threadIdx.x == 0) *wide_flag = 1;
    return;
  }
  if (path == 0) {
    if (threadIdx.x < 32) regwin_factor(n, kl, ku, AB, (int)ldab, ipiv, d_info);
  } else if (path == 1) {
    if (K == 1) window_factor_pf<1>(PF, n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
    else if (K == 2) window_factor_pf<2>(PF, n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
    else if (K == 4) window_factor_pf<4>(PF, n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
    else window_factor_pf<8>(PF, n, kl, ku, AB, ldab, ipiv, d_info, W, sh);
  } else {
    generic_factor(n, kl, ku, AB, ldab, ipiv, d_info);
  }
}

template <int K, int PF>
int launch_window(long long n, int kl, int ku, double *AB, long long ldab, int *ipiv, int *d_info, size_t smem,
                  cudaStream_t s) {
  if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_gbtrf_window<K, PF>), 200 * 1024)) return BANDLU_ERR_CUDA;
  k_gbtrf_window<K, PF><<<1, kWarps * 32, smem, s>>>((int)n, kl, ku, AB, ldab, ipiv, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

template <int K>
int launch_window_pf(int pf, long long n, int kl, int ku, double *AB, long long ldab, int *ipiv, int *d_info,
                     size_t smem, cudaStream_t s) {
  if (pf <= 1) return launch_window<K, 1>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
  if (pf <= 2) return launch_window<K, 2>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
  if (pf <= 4) return launch_window<K, 4>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
  return launch_window<K, 8>(n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
}

}  // namespace

int launch_gbtrf(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t s,
                 bool allow_alloc) {
  if (n == 0) {
    if (cudaMemsetAsync(d_info, 0, sizeof(int), s) != cudaSuccess) return BANDLU_ERR_CUDA;
    return BANDLU_OK;
  }
  int K = 1, PF = 1;
  size_t smem = 0;
  const int path = factor_path(n, kl, ku, ldab, &K, &PF, &smem);
  if (path == 0) {
    k_gbtrf_regwin<<<1, 32, 0, s>>>((int)n, kl, ku, AB, (int)ldab, ipiv, d_info);
    BANDLU_CHECK_LAUNCH();
    return BANDLU_OK;
  }
  if (path == 1) {
    if (K == 1) return launch_window_pf<1>(PF, n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
    if (K == 2) return launch_window_pf<2>(PF, n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
    if (K == 4) return launch_window_pf<4>(PF, n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
    return launch_window_pf<8>(PF, n, kl, ku, AB, ldab, ipiv, d_info, smem, s);
  }
  if (allow_alloc) {
    bool used = false;
    const int rc = launch_gbtrf_wide(n, kl, ku, AB, ldab, ipiv, d_info, s, &used);
    if (rc != BANDLU_OK || used) return rc;
  }
  k_gbtrf_generic<<<1, 1024, 0, s>>>(n, kl, ku, AB, ldab, ipiv, d_info);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu

namespace bandlu {

int launch_gbtrf_on_device(int64_t n, double *AB, int64_t ldab, int *ipiv, const int *d_kl, const int *d_ku,
                           const int *d_status, int *d_info, cudaStream_t s) {
  if (n == 0) return BANDLU_OK;
  // every shared-memory window that fits the band storage: kl <= kWinMaxKl and
  // CS = 2*kl+ku+1 <= min(ldab, 256) column slots of R = kl+1+kDelta rows
  const long long cs = ldab < 256 ? ldab : 256;
  const size_t smem = (size_t)((kWinMaxKl + 1 + kDelta) * cs) * sizeof(double);
  if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_gbtrf_on_device), 200 * 1024)) return BANDLU_ERR_CUDA;
  // a band storage that admits kl >= kWinMaxKl + 1 may hold a band no window takes:
  // the multi-CTA kernel is enqueued too and runs only if the decision on the device is its
  WideDeferred wd;
  if (ldab >= 2 * (kWinMaxKl + 1) + 1) {
    const int rc = prepare_gbtrf_wide_deferred(n, ldab, s, &wd);
    if (rc != BANDLU_OK) return rc;
  }
  k_gbtrf_on_device<<<1, kWarps * 32, smem, s>>>((int)n, AB, ldab, ipiv, d_kl, d_ku, d_status, d_info, smem,
                                                 wd.rows_cap, wd.flags != nullptr ? wd.flags + 1 : nullptr);
  if (cudaPeekAtLastError() != cudaSuccess) {
    if (wd.flags != nullptr) cudaFreeAsync(wd.flags, s);
    return BANDLU_ERR_CUDA;
  }
  if (wd.rows_cap > 0) return launch_gbtrf_wide_deferred(wd, n, AB, ldab, ipiv, d_kl, d_ku, d_info, s);
  return BANDLU_OK;
}

}  // namespace bandlu
