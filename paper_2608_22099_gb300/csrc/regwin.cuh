// regwin.cuh -- banded LU with the active window in registers, for bands whose
// window (kl+1) x (kl+ku+1) fits a warp (Sec. II-A step 3; f(N) ~ O(N*P*Q),
// Eq. S-N-N3).  Used by the single-matrix gbtrf for the narrowest bands and by
// the batched factorisation.
#pragma once

#include "common.cuh"
#include "rcp.cuh"

namespace bandlu {
namespace regwin {

// warp_argmax_first_z without its shortcut: both reductions, always.  Several
// segments' argmaxes in a row (S > 1), and the windowed kernel's panel warp, run
// faster without the shortcut's branch (measured).
__device__ __forceinline__ int argmax_two_pass(unsigned long long key, bool *all_zero) {
  const unsigned hi = (unsigned)(key >> 32), lo = (unsigned)key;
  const unsigned mhi = __reduce_max_sync(FULL, hi);
  const unsigned lo2 = (hi == mhi) ? lo : 0u;
  const unsigned mlo = __reduce_max_sync(FULL, lo2);
  const unsigned win = __ballot_sync(FULL, hi == mhi && lo == mlo);
  *all_zero = (mhi | mlo) == 0u;
  return __ffs(win) - 1;
}

constexpr int kWinPrefetch = 8;  // entering rows a window keeps in flight

// Banded elimination with the active window in registers, in place on band
// storage (ldab x n).  It reads only the band's own entries and writes U's rows
// and the multipliers; fill-row entries above the matrix, which no step
// writes, are the caller's (the elimination clears them).  The warp is cut into S
// segments of W = 32/S lanes; segment s factors its own matrix (ab[s], kl[s],
// ku[s], ipiv[s]), all of the same order n, with (kl+1)*(kl+ku+1) <= W.  Every
// warp instruction thus serves S matrices.
//
// At step j a segment's window holds rows j..j+kl and columns j..j+kv
// (kv = kl+ku), element (r, c) on segment lane r*C + c (C = kv+1).  Step j:
// first-max argmax over column 0, interchange of rows 0 and p (whole window
// rows: beyond the running reach ju both entries are zero fill), multipliers,
// rank-1 update with the zero-u skip, then row 0 (U row j) and column 0 below
// it (multipliers) are written to their places in AB and the window moves one
// step down the diagonal: entries shift up and left, the entering column holds
// structural zeros (no earlier step reached it), and the entering row j+1+kl
// is the untouched original row, read kWinPrefetch steps ahead.  Every AB
// entry a step writes belongs to a row that entered the window earlier, so
// reading and writing in place do not collide; the fill rows are never read
// (the window holds their zeros).  Same operations in the same order as the
// unblocked elimination: the factors are bit-identical to it.
// 32-bit offsets: requires (n+1) * ldab < 2^31.
template <int S>
__device__ __forceinline__ void window_gbtrf(double *const (&abs)[S], int ldab, int n, const int (&kls)[S], const int (&kus)[S],
                             int *const (&ipivs)[S], int (&infos)[S]) {
  constexpr int W = 32 / S;
  const int lane = threadIdx.x & 31;
  const int seg = lane / W, sl = lane - seg * W, base = seg * W;
  int kl = kls[0], ku = kus[0];
  double *ab = abs[0];
  int *ipiv = ipivs[0];
#pragma unroll
  for (int t = 1; t < S; ++t)
    if (seg == t) {
      kl = kls[t];
      ku = kus[t];
      ab = abs[t];
      ipiv = ipivs[t];
    }
  const int kv = kl + ku, C = kv + 1, L = kl + 1;
  const bool inw = sl < L * C;
  const int r = inw ? sl / C : 0, c = inw ? sl - r * C : 0;
  const bool feeder = inw && r == kl;  // lanes of the entering row
  // row i's element in column i-kl+c sits at AB(kv+kl-c, i-kl+c), always inside
  // the band's diagonals
  const int feed_off = (kv + kl - c) + (c - kl) * ldab;  // + i * ldab
  const int ushift = (kv - c) + c * ldab;                 // U(j, j+c): + j * ldab
  const int lshift = kv + r;                              // l_{j+r, j}: + j * ldab
  double w = 0.0;
  if (inw && r < n && c < n && c - r <= ku && r - c <= kl) w = __ldcg(ab + (kv + r - c) + c * ldab);
  // q[s] holds the entering row of the next step j with j % kWinPrefetch == s
  // (row j+1+kl, columns j+1+c); it is refilled kWinPrefetch steps ahead.  The
  // step loop is unrolled by kWinPrefetch so that every slot is one register
  // (rotating the slots would wait on each load a step after issuing it).
  double q[kWinPrefetch];
#pragma unroll
  for (int k = 0; k < kWinPrefetch; ++k) {
    const int i = kl + 1 + k;
    q[k] = (feeder && i < n && i - kl + c < n) ? __ldcg(ab + feed_off + i * ldab) : 0.0;
  }
  int info = 0;
  int piv_acc = 0;  // segment lane t keeps ipiv of step W*m + t until the block of W is stored
  for (int j0 = 0; j0 < n; j0 += kWinPrefetch) {
#pragma unroll
    for (int sidx = 0; sidx < kWinPrefetch; ++sidx) {
      const int j = j0 + sidx;
      if (j >= n) break;
      const int km = min(kl, n - 1 - j);
      const bool cand = inw && c == 0 && r <= km;
      bool myspec;
      const double myr = rcp_rn_fast(w, &myspec);
      const unsigned long long key = cand ? pivot_abs_key(w, r == 0) : 0ull;
      int win = 0;
      bool zp = false;  // exact zero pivot (then p == 0)
#pragma unroll
      for (int t = 0; t < S; ++t) {
        bool allz;
        const int wt = S == 1 ? warp_argmax_first_z(key, &allz) : argmax_two_pass(seg == t ? key : 0ull, &allz);
        if (seg == t) {
          win = wt;
          zp = allz;
        }
      }
      const int p = __shfl_sync(FULL, r, win);
      double rc = __shfl_sync(FULL, myr, win);
      const bool spec = __shfl_sync(FULL, myspec ? 1 : 0, win) != 0;
      const double pv = __shfl_sync(FULL, w, win);
      if (__any_sync(FULL, spec && !zp) && spec && !zp) rc = rcp_division(pv);
      // interchange rows 0 and p
      const int src = (r == 0) ? win + c : ((r == p) ? base + c : lane);
      w = __shfl_sync(FULL, w, src);
      const bool below = inw && r >= 1 && r <= km;
      if (!zp && below && c == 0) w = w * rc;              // multiplier l_{j+r, j}
      const double u = __shfl_sync(FULL, w, base + c);     // row 0 (U row j), column c
      const double l = __shfl_sync(FULL, w, lane - c);     // multiplier of row r
      if (!zp && below && c >= 1) {
        const double t = fma(-l, u, w);
        w = nz(u) ? t : w;
      }
      // U(j, j+c) -> AB(kv-c, j+c); l_{j+r, j} -> AB(kv+r, j)
      if (inw && r == 0 && j + c < n) ab[ushift + j * ldab] = w;
      if (inw && c == 0 && r >= 1 && r <= km) ab[lshift + j * ldab] = w;
      if (sl == j % W) piv_acc = j + p + 1;
      if (j % W == W - 1 || j == n - 1) {
        if (sl <= j % W) ipiv[j - j % W + sl] = piv_acc;
      }
      if (zp && info == 0) info = j + 1;
      // move the window one step down the diagonal
      const double sh = __shfl_sync(FULL, w, base + ((sl + C + 1) & (W - 1)));
      w = (r < kl) ? ((c < kv) ? sh : 0.0) : q[sidx];
      const int i = j + 1 + kl + kWinPrefetch;
      q[sidx] = (feeder && i < n && i - kl + c < n) ? __ldcg(ab + feed_off + i * ldab) : 0.0;
    }
  }
#pragma unroll
  for (int t = 0; t < S; ++t) infos[t] = __shfl_sync(FULL, info, t * W);
}

}  // namespace regwin
}  // namespace bandlu
