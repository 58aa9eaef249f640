// trwin.cuh -- one sweep of a banded triangular solve by one warp, with the
// active part of the right-hand side in registers.  Both halves of the band
// solve after gbtrf (xGBTRS) and the banded triangular solves of the dispatch
// (xTBSV, no transpose) are such sweeps.
//
// A sweep visits positions k = 0..n-1 (row k going forward, row n-1-k going
// backward).  Step k, with x the value at position k:
//   kPiv: x and the value at position k + p_k are interchanged first;
//   if x != 0 (the reference-BLAS zero test):
//     kDiv: x = x / c(k, 0)               (IEEE quotient: div_known, with the
//                                         reciprocals formed 32 steps at a time)
//     position k + t takes fma(-c(k, t), x, .) for t = 1..min(kw, n-1-k);
//   x is final and is stored.
// c(k, t) is the coefficient at the source functor's address at(k, t) (t = 0:
// the divisor).
//
// Layout: a window of W = 32*RW positions k..k+W-1 that ROTATES instead of
// shifting: position m lives on lane m % 32, register (m / 32) % RW, for as
// long as it is in the window.  A finished position's slot takes the position
// W further on.  A step therefore moves no data between lanes except the one
// broadcast of x (and the two values of an interchange), and the FP64 update
// skips every register that holds no position k+1..k+mk.  Each lane loads the
// coefficients of the positions it holds kPf steps ahead into registers (the
// step loop is unrolled by kPf, one register per slot), as predicated loads
// that nothing consumes before their step.  (Measured on GB300: a per-warp
// shared-memory ring filled by cp.async, waited on one commit group per step,
// made every step slower than these register loads do.)
#pragma once

#include "common.cuh"
#include "rcp.cuh"

namespace bandlu {
namespace trwin {

// Coefficients of the sweeps.  k is the step; t >= 0 the offset from the
// eliminated position.
// at(k, t): the coefficient's address.  prefetch(k, kw, n, lane): called once
// per step k by every lane, asks L2 for data the sweep reads kPrefetchSteps
// steps later (a no-op for the band storage, which the factorisation has just
// left in L2).
constexpr int kPrefetchSteps = 48;

struct GbLower {  // forward half of xGBTRS: multipliers l_{k+t,k} = AB(kv+t, k)
  const double *AB;
  int ldab, kv;
  __device__ __forceinline__ const double *at(int k, int t) const { return AB + (kv + t) + (long long)k * ldab; }
  __device__ __forceinline__ void prefetch(int, int, int, int) const {}
};
struct GbUpper {  // backward half of xGBTRS: j = n-1-k, U(j-t, j) = AB(kv-t, j)
  const double *AB;
  int ldab, kv, n;
  __device__ __forceinline__ const double *at(int k, int t) const {
    return AB + (kv - t) + (long long)(n - 1 - k) * ldab;
  }
  __device__ __forceinline__ void prefetch(int, int, int, int) const {}
};
// In the dense matrix the coefficients of one step lie in different rows (one
// 32-byte sector each), but row m's band segment -- used over kw consecutive
// steps -- is contiguous: lane L prefetches the L-th 128-byte line of the
// segment of the row whose first use is kPrefetchSteps steps ahead.
__device__ __forceinline__ void prefetch_l2_line(const double *p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
struct DenseLower {  // lower triangular, row-major dense: L(k+t, k) = A[(k+t)*lda + k]
  const double *A;
  long long lda;
  __device__ __forceinline__ const double *at(int k, int t) const { return A + (long long)(k + t) * lda + k; }
  // row m = k + kw + kPrefetchSteps is first read at step m - kw; its segment is
  // A[m*lda + m-kw .. m-1]
  __device__ __forceinline__ void prefetch(int k, int kw, int n, int lane) const {
    const int m = k + kw + kPrefetchSteps;
    if (m < n && lane * 16 < kw) prefetch_l2_line(A + (long long)m * lda + (m - kw) + lane * 16);
  }
};
struct DenseUpper {  // upper triangular, row-major dense: j = n-1-k, U(j-t, j) = A[(j-t)*lda + j]
  const double *A;
  long long lda;
  int n;
  __device__ __forceinline__ const double *at(int k, int t) const {
    const int j = n - 1 - k;
    return A + (long long)(j - t) * lda + j;
  }
  // row m = j - kw - kPrefetchSteps is first read at column m + kw; its segment
  // is A[m*lda + m+1 .. m+kw]
  __device__ __forceinline__ void prefetch(int k, int kw, int, int lane) const {
    const int m = n - 1 - k - kw - kPrefetchSteps;
    if (m >= 0 && lane * 16 < kw) prefetch_l2_line(A + (long long)m * lda + (m + 1) + lane * 16);
  }
};

// *p where c holds, else 0.0, as one predicated load: a load followed by a
// select would make the select (and so the step that issues the read-ahead)
// wait for the data.  ld_coef reads through the read-only path (coefficients);
// ld_rhs through the ordinary one (the right-hand side, which the sweep writes).
__device__ __forceinline__ double ld_coef(const double *p, bool c) {
  double v;
  asm("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %2, 0;\n\tmov.b64 %0, 0;\n\t@q ld.global.nc.f64 %0, [%1];\n\t}"
      : "=d"(v)
      : "l"(p), "r"((unsigned)c));
  return v;
}
__device__ __forceinline__ double ld_rhs(const double *p, bool c) {
  double v;
  // (never an entry the sweep has written: positions are read once, before their step)
  asm("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %2, 0;\n\tmov.b64 %0, 0;\n\t@q ld.global.f64 %0, [%1];\n\t}"
      : "=d"(v)
      : "l"(p), "r"((unsigned)c));
  return v;
}

// Value at window position m, broadcast to every lane.
template <int RW>
__device__ __forceinline__ double get(const double (&w)[RW], int m) {
  const int rr = (m >> 5) & (RW - 1);
  double v = w[0];
#pragma unroll
  for (int r = 1; r < RW; ++r) v = dsel(rr == r, w[r], v);
  return __shfl_sync(FULL, v, m & 31);
}

template <int RW>
__device__ __forceinline__ void put(double (&w)[RW], int m, double v, int lane) {
  const int rr = (m >> 5) & (RW - 1);
  const bool mine = lane == (m & 31);
#pragma unroll
  for (int r = 0; r < RW; ++r) w[r] = dsel(mine && rr == r, v, w[r]);
}

// The sweep.  b: the right-hand side (n doubles, overwritten with the result);
// kw: the band width of the update (kl or kl+ku); ipiv (kPiv only): 1-based
// interchanges of the forward half of xGBTRS, position k with ipiv[k]-1.
template <int RW, int kPf, bool kFwd, bool kPiv, bool kDiv, class Src>
__device__ __forceinline__ void sweep(double *b, int n, int kw, const Src &src, const int *ipiv) {
  constexpr int W = 32 * RW;
  const int lane = threadIdx.x & 31;
  auto row = [&](int m) { return kFwd ? m : n - 1 - m; };
  // offset from step k of the position this lane holds in register r
  auto off = [&](int k, int r) { return (lane + 32 * r - k) & (W - 1); };

  double w[RW];
#pragma unroll
  for (int r = 0; r < RW; ++r) {
    const int m = lane + 32 * r;
    w[r] = ld_rhs(b + row(m), m < n);
  }
  // slot s: coefficients of step k0+s for the positions this lane holds, the
  // value entering the window after that step (its owner lane only), the
  // interchange and the divisor
  double cf[kPf][RW], en[kPf];
  int pv[kPf];
  auto fill = [&](int s, int k) {
    const int mk = min(kw, n - 1 - k);  // negative past the end: no coefficient
#pragma unroll
    for (int r = 0; r < RW; ++r) {
      const int t = off(k, r);
      cf[s][r] = ld_coef(src.at(k, t), t >= 1 && t <= mk);
    }
    en[s] = ld_rhs(b + row(k + W), lane == (k & 31) && k + W < n);
    // the raw entry (a clamped index, no select): nothing may consume a load
    // before the step that needs it
    if (kPiv) pv[s] = __ldg(ipiv + min(k, n - 1));
  };
#pragma unroll
  for (int s = 0; s < kPf; ++s) fill(s, s);

  // divisors, 32 steps at a time: lane L holds the divisor of step 32*B + L of
  // the current block B with its two-term reciprocal (div_known_prep), formed
  // in parallel once per block; the next block's divisors are read a block ahead
  double bd = 1.0, byh = 1.0, byl = 0.0, nd = 1.0;
  bool bok = true;
  if (kDiv) nd = __ldg(src.at(min(lane, n - 1), 0));  // steps past the end read a valid dummy
  for (int k0 = 0; k0 < n; k0 += kPf) {
#pragma unroll
    for (int s = 0; s < kPf; ++s) {
      const int k = k0 + s;
      if (k >= n) break;
      const int mk = min(kw, n - 1 - k);
      double dj = 1.0, yhj = 1.0, ylj = 0.0;
      bool okj = true;
      if (kDiv) {
        if ((k & 31) == 0) {  // uniform: a new block of 32 steps
          bd = nd;
          nd = __ldg(src.at(min(k + 32 + lane, n - 1), 0));
          div_known_prep(bd, &byh, &byl, &bok);
        }
        dj = __shfl_sync(FULL, bd, k & 31);
        yhj = __shfl_sync(FULL, byh, k & 31);
        ylj = __shfl_sync(FULL, byl, k & 31);
        okj = __shfl_sync(FULL, (int)bok, k & 31) != 0;
      }
      if (kPiv) {
        int p = pv[s] - 1 - k;
        if (p < 0 || p > mk) p = 0;  // past the end, or outside the window: ignored
        if (p != 0) {  // uniform
          const double a = get(w, k), c = get(w, k + p);
          put(w, k, c, lane);
          put(w, k + p, a, lane);
        }
      }
      double x = get(w, k);
      if (nz(x)) {  // uniform
        if (kDiv) x = div_known(x, dj, yhj, ylj, okj);
        // registers holding positions k+1..k+mk: the 32-position chunks c0..c1
        const int c0 = (k + 1) >> 5, c1 = (k + mk) >> 5;
#pragma unroll
        for (int r = 0; r < RW; ++r) {
          if (mk >= 1 && ((r - c0) & (RW - 1)) <= c1 - c0) {  // uniform
            const int t = off(k, r);
            const double u = fma(-cf[s][r], x, w[r]);
            w[r] = dsel(t >= 1 && t <= mk, u, w[r]);
          }
        }
      }
      if (lane == (k & 31)) b[row(k)] = x;
      put(w, k, en[s], lane);  // position k leaves, position k+W enters
      fill(s, k + kPf);
      src.prefetch(k, kw, n, lane);
    }
  }
}

}  // namespace trwin
}  // namespace bandlu
