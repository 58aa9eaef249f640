// gbtrs.cu -- the solve after the factorisation: the backslash operator that the
// dispatch of Listing 1 stands for (Sec. I-A; LAPACK xGBTRS, no transpose).
//
// A X = B with A = P0 L0 P1 L1 ... U as left by gbtrf.  Each right-hand side is
// two chains of n dependent steps:
//   forward  j = 0..n-2: interchange b_j and b_{ipiv_j}; if b_j != 0, rows
//            j+1..j+kl take fma(-l, b_j, .);
//   backward j = n-1..0: if b_j != 0, b_j = b_j / u_jj and rows j-kv..j-1 take
//            fma(-b_j, u, .).
// The active part of b stays in registers, in a window that rotates with the
// steps: one warp per right-hand side up to kl+ku+1 = 128 rows (trwin.cuh), a
// CTA of 256 or 512 threads per right-hand side and sweep above (cta_sweep).
// The division by u_jj uses a two-term reciprocal formed ahead of time
// (div_known: four dependent FP64 operations instead of a full division).  The
// same operations in the same order as the oracle, so the solution is
// bit-identical to it.  Interchanges outside j..j+kl (not produced by gbtrf)
// are ignored.
#include <climits>
#include <cstdlib>

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

// ---------------------------------------------------------------------------
// Wide windows: one CTA of NT threads per right-hand side runs a sweep with the
// active part of b in registers.  Position m lives on thread m % NT, register
// (m / NT) % R, for as long as it is in the window of W = NT*R positions: the
// rotating window of trwin.cuh, spread over the CTA's warps.  A step costs one
// barrier.
//   Before it, the owners of what step k reads publish it in shared memory:
//   forward, the value at position k and the one it is interchanged with;
//   backward, the quotient x_k, which its owner forms (div_known_nz, the
//   divisor's two-term reciprocal ready) right after applying step k-1 to that
//   position, before the other registers of its warp.
//   After it, every thread applies step k to the positions k+1..k+mk it holds:
//   one FP64 instruction per warp register that holds any of them, with the
//   zero test as a select after it.  Everything that does not depend on the
//   step's value is computed before the barrier.
// The warp whose 32 positions a block of 32 steps eliminates refills them at the
// block's end with the positions W further on (W >= kw + 33, so a refilled
// position is first updated after that block).  The divisors of a block are read
// two blocks ahead and given their reciprocals one block ahead, by the warp that
// will own them; coefficients are read kPf steps ahead into registers, and the
// band column of step k + kCtaL2Ahead is requested into L2 (the band of a wide
// factorisation does not stay in L2).  Same operations, same order as the sweep
// of trwin.cuh and the oracle.
constexpr int kCtaL2Ahead = 48;

template <int R>
__device__ __forceinline__ double reg_get(const double (&w)[R], int r) {
  double v = w[0];
#pragma unroll
  for (int i = 1; i < R; ++i) v = dsel(r == i, w[i], v);
  return v;
}
template <int R>
__device__ __forceinline__ void reg_set(double (&w)[R], int r, double v) {
#pragma unroll
  for (int i = 0; i < R; ++i) w[i] = dsel(r == i, v, w[i]);
}

// Lowest address and length (doubles) of the coefficients step k reads: the
// multipliers AB(kv+1..kv+mk, k), or U(j-mk..j, j) = AB(kv-mk..kv, j), j = n-1-k.
__device__ __forceinline__ const double *band_segment(const trwin::GbLower &s, int k, int mk, int *len) {
  *len = mk;
  return s.at(k, 1);
}
__device__ __forceinline__ const double *band_segment(const trwin::GbUpper &s, int k, int mk, int *len) {
  *len = mk + 1;
  return s.at(k, mk);
}

template <int NT, int R, int kPf, bool kFwd, bool kPiv, bool kDiv, class Src>
__device__ __forceinline__ void cta_sweep(double *b, int n, int kw, const Src &src, const int *ipiv, double *pub) {
  constexpr int W = NT * R, NWARP = NT / 32, NQ = W / 32;
  static_assert((NT & (NT - 1)) == 0 && NWARP >= 3 && kPf >= 2, "window layout");
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  auto row = [&](int m) { return kFwd ? m : n - 1 - m; };
  auto off = [&](int k, int r) { return (tid + NT * r - k) & (W - 1); };  // offset of the position in register r
  auto mk_of = [&](int k) { return min(kw, n - 1 - k); };
  auto owner = [&](int m) { return m & (NT - 1); };
  auto reg_of = [&](int m) { return (m / NT) & (R - 1); };
  auto bw = [&](int B) { return B & (NWARP - 1); };  // the warp that holds the positions of block B
  auto piv_off = [&](int k, int raw) {               // interchange offset; outside the window: ignored
    const int p = raw - 1 - k;
    return (p < 0 || p > mk_of(k)) ? 0 : p;
  };

  double w[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int m = tid + NT * r;
    w[r] = trwin::ld_rhs(b + row(m), m < n);
  }
  double cf[kPf][R];
  int pv[kPf];
  auto fill = [&](int s, int k) {
    const int mk = mk_of(k);  // negative past the end: no coefficient
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int t = off(k, r);
      cf[s][r] = trwin::ld_coef(src.at(k, t), t >= 1 && t <= mk);
    }
    if (kPiv) pv[s] = __ldg(ipiv + min(k, n - 1));
  };
#pragma unroll
  for (int s = 0; s < kPf; ++s) fill(s, s);

  // divisors: lane L of warp bw(B) holds that of position 32B + L (bd) with its
  // two-term reciprocal while block B runs; nd is the next block it will own
  double nd = 1.0, bd = 1.0, byh = 1.0, byl = 0.0, en = 0.0;
  bool bok = true;
  auto dload = [&](int B) { return __ldg(src.at(min(32 * B + lane, n - 1), 0)); };
  if (kDiv) {
    if (warp == bw(0)) {
      bd = dload(0);
      div_known_prep(bd, &byh, &byl, &bok);
    }
    if (warp == bw(1)) nd = dload(1);
  }
  // What step k reads, published by its owners into slot k & 1 of pub (value,
  // interchange partner): here step 0's, before the loop; inside it, each step
  // publishes for the next.
  auto publish = [&](int k, int s) {
    if (kDiv) {
      if (warp == (owner(k) >> 5) && lane == (k & 31)) {
        const double x = div_known_nz(reg_get(w, reg_of(k)), bd, byh, byl, bok);
        pub[(k & 1) * 2] = x;
        b[row(k)] = x;
      }
    } else {
      if (tid == owner(k)) pub[(k & 1) * 2] = reg_get(w, reg_of(k));
      if (kPiv) {
        const int p = piv_off(k, pv[s]);
        if (p != 0 && tid == owner(k + p)) pub[(k & 1) * 2 + 1] = reg_get(w, reg_of(k + p));
      }
    }
  };
  if (n > 0) publish(0, 0);

  for (int k0 = 0; k0 < n; k0 += kPf) {
#pragma unroll
    for (int s = 0; s < kPf; ++s) {
      const int k = k0 + s;
      if (k >= n) break;  // uniform
      // what does not depend on the step's value, ahead of the barrier
      const int mk = mk_of(k);
      const int c0 = (k + 1) >> 5, c1 = (k + mk) >> 5;
      bool cin[R], tin[R];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        cin[r] = mk >= 1 && (((warp + NWARP * r) - c0) & (NQ - 1)) <= c1 - c0;  // uniform: a position in range
        const int t = off(k, r);
        tin[r] = t >= 1 && t <= mk;
      }
      const int k1 = k + 1;
      const int s1 = (s + 1) % kPf;
      const bool crit = k1 < n && warp == (owner(k1) >> 5);  // this warp publishes for step k+1
      const int rr = reg_of(k1);
      const bool k1own = k1 < n && tid == owner(k1);
      int p = 0, pr = 0, p1r = 0;
      bool pown = false, p1own = false;
      if (kPiv) {
        p = piv_off(k, pv[s]);
        pown = p != 0 && tid == owner(k + p);
        pr = reg_of(k + p);
        const int p1 = k1 < n ? piv_off(k1, pv[s1]) : 0;
        p1own = p1 != 0 && tid == owner(k1 + p1);
        p1r = reg_of(k1 + p1);
      }
      __syncthreads();  // step k's values are published
      double x = pub[(k & 1) * 2];
      if (kPiv && p != 0) {  // uniform
        const double c = pub[(k & 1) * 2 + 1];
        if (pown) reg_set(w, pr, x);
        x = c;
      }
      const bool go = nz(x);  // the zero test: a select after the multiply-add, off the chain
      auto upd = [&](int r) {  // step k on the positions register r holds in k+1..k+mk
        if (cin[r]) {          // uniform
          const double u = fma(-cf[s][r], x, w[r]);
          w[r] = dsel(go && tin[r], u, w[r]);
        }
      };
      if (crit) {  // the register holding position k+1 first, then what step k+1 reads
#pragma unroll
        for (int r = 0; r < R; ++r)
          if (r == rr) upd(r);
        if (k1own) {
          if (kDiv) {
            const double q = div_known_nz(reg_get(w, rr), bd, byh, byl, bok);
            pub[(k1 & 1) * 2] = q;
            b[row(k1)] = q;
          } else {
            pub[(k1 & 1) * 2] = reg_get(w, rr);
          }
        }
#pragma unroll
        for (int r = 0; r < R; ++r)
          if (r != rr) upd(r);
      } else {
#pragma unroll
        for (int r = 0; r < R; ++r) upd(r);
      }
      if (kPiv && p1own) pub[(k1 & 1) * 2 + 1] = reg_get(w, p1r);  // step k+1's interchange partner
      if (!kDiv && tid == owner(k)) b[row(k)] = x;  // final (a quotient was stored by its owner)
      if ((k & 31) == 0) {  // block B starts (uniform)
        const int B = k >> 5;
        if (warp == bw(B)) en = trwin::ld_rhs(b + row(k + W + lane), k + W + lane < n);
        if (kDiv) {
          if (warp == bw(B + 1)) {
            bd = nd;
            div_known_prep(bd, &byh, &byl, &bok);
          }
          if (warp == bw(B + 2)) nd = dload(B + 2);
        }
      }
      if ((k & 31) == 31 && warp == bw(k >> 5)) reg_set(w, reg_of(k), en);  // its positions leave, W on enter
      fill(s, k + kPf);
      {
        const int kp = k + kCtaL2Ahead;
        if (kp < n && warp == bw((k >> 5) + NWARP / 2)) {
          int len;
          const double *a0 = band_segment(src, kp, mk_of(kp), &len);
          for (int i = lane * 16; i < len; i += 32 * 16) trwin::prefetch_l2_line(a0 + i);
        }
      }
    }
  }
}

template <int NT, int R, int kPf>
__global__ void __launch_bounds__(NT, 1)
    k_gbtrs_wide_fwd(int n, int kl, int ku, const double *__restrict__ AB, int ldab, const int *__restrict__ ipiv,
                     double *__restrict__ B, long long ldb, const int *__restrict__ d_info) {
  __shared__ double pub[4];
  if (d_info != nullptr && *d_info != 0) return;  // a singular factor: B is left as it is
  cta_sweep<NT, R, kPf, true, true, false>(B + (long long)blockIdx.x * ldb, n, kl, trwin::GbLower{AB, ldab, kl + ku},
                                       ipiv, pub);
}

template <int NT, int R, int kPf>
__global__ void __launch_bounds__(NT, 1)
    k_gbtrs_wide_bwd(int n, int kl, int ku, const double *__restrict__ AB, int ldab, double *__restrict__ B,
                     long long ldb, const int *__restrict__ d_info) {
  __shared__ double pub[4];
  if (d_info != nullptr && *d_info != 0) return;
  const int kv = kl + ku;
  cta_sweep<NT, R, kPf, false, false, true>(B + (long long)blockIdx.x * ldb, n, kv, trwin::GbUpper{AB, ldab, kv, n},
                                        nullptr, pub);
}

// Registers per thread for a window of W = NT*R >= kw + 33 positions (0: too wide).
constexpr int cta_regs(long long kw, int NT, int rmax) {
  return kw + 33 <= NT ? 1 : (kw + 33 <= 2LL * NT ? 2 : (kw + 33 <= 4LL * NT && rmax >= 4 ? 4 : 0));
}

template <int NT>
void launch_fwd_nt(int n, int kl, int ku, int nrhs, const double *AB, int ldab, const int *ipiv, double *B,
                   long long ldb, const int *d_info, cudaStream_t s) {
  constexpr int kPf = 8, rmax = NT >= 512 ? 2 : 4;  // registers: 8 coefficients per window register and thread
  const int r = cta_regs(kl, NT, rmax);
  if (r == 1)
    k_gbtrs_wide_fwd<NT, 1, kPf><<<(unsigned)nrhs, NT, 0, s>>>(n, kl, ku, AB, ldab, ipiv, B, ldb, d_info);
  else if (r == 2)
    k_gbtrs_wide_fwd<NT, 2, kPf><<<(unsigned)nrhs, NT, 0, s>>>(n, kl, ku, AB, ldab, ipiv, B, ldb, d_info);
  else
    k_gbtrs_wide_fwd<NT, rmax, kPf><<<(unsigned)nrhs, NT, 0, s>>>(n, kl, ku, AB, ldab, ipiv, B, ldb, d_info);
}

template <int NT>
void launch_bwd_nt(int n, int kl, int ku, int nrhs, const double *AB, int ldab, double *B, long long ldb,
                   const int *d_info, cudaStream_t s) {
  constexpr int kPf = 8, rmax = NT >= 512 ? 2 : 4;
  const int r = cta_regs((long long)kl + ku, NT, rmax);
  if (r == 1)
    k_gbtrs_wide_bwd<NT, 1, kPf><<<(unsigned)nrhs, NT, 0, s>>>(n, kl, ku, AB, ldab, B, ldb, d_info);
  else if (r == 2)
    k_gbtrs_wide_bwd<NT, 2, kPf><<<(unsigned)nrhs, NT, 0, s>>>(n, kl, ku, AB, ldab, B, ldb, d_info);
  else
    k_gbtrs_wide_bwd<NT, rmax, kPf><<<(unsigned)nrhs, NT, 0, s>>>(n, kl, ku, AB, ldab, B, ldb, d_info);
}

// Threads of a sweep's CTA: the smallest CTA that holds the window with one
// register per thread (measured on GB300, kl = ku = 64: 256 threads 622 ns per
// row, 512 threads 696; kl = ku = 128: 512 threads with one register 716 ns per
// row, 256 threads with two 857), else 512 threads with two registers (R = 4 on
// 256 threads was slower still).  BANDLU_GBTRS_CTA_THREADS=256|512 forces one
// size, for measurement.
int cta_threads(long long kw) {
  static const int forced = [] {
    const char *v = std::getenv("BANDLU_GBTRS_CTA_THREADS");
    const int t = v != nullptr ? std::atoi(v) : 0;
    return (t == 256 || t == 512) ? t : 0;
  }();
  if (forced) return forced;
  return kw + 33 <= 256 ? 256 : 512;
}

bool wide_fits(long long kv) { return cta_regs(kv, cta_threads(kv), cta_threads(kv) >= 512 ? 2 : 4) > 0; }

int launch_wide(int n, int kl, int ku, int nrhs, const double *AB, int ldab, const int *ipiv, double *B,
                long long ldb, const int *d_info, cudaStream_t s) {
  if (kl > 0 && n > 1) {
    if (cta_threads(kl) == 256)
      launch_fwd_nt<256>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    else
      launch_fwd_nt<512>(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, s);
    BANDLU_CHECK_LAUNCH();
  }
  const long long kv = (long long)kl + ku;
  if (cta_threads(kv) == 256)
    launch_bwd_nt<256>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  else
    launch_bwd_nt<512>(n, kl, ku, nrhs, AB, ldab, B, ldb, d_info, s);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
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

// Windows up to this many rows take the one-warp register window, wider ones the
// CTA-wide window (measured on GB300, n = 16384: the CTA 1.9x faster at kl+ku+1 =
// 129 and 2.4x at 451; the one-warp window faster at 65 and 73 than the first,
// 512-thread CTA; BANDLU_GBTRS_CTA_ABOVE=<rows> moves the switch, for measurement).
long long cta_min_window() {
  static const long long w = [] {
    const char *v = std::getenv("BANDLU_GBTRS_CTA_ABOVE");
    return v != nullptr ? std::atoll(v) : 128LL;
  }();
  return w;
}

}  // namespace

int launch_gbtrs(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
                 int64_t ldb, const int *d_info, cudaStream_t s) {
  if (n == 0 || nrhs == 0) return BANDLU_OK;
  const long long win = (long long)kl + ku + 1;  // rows the backward window needs (>= kl + 1)
  if (n <= INT_MAX / 2 && ldab <= INT_MAX && nrhs <= INT_MAX) {
    if (win <= cta_min_window()) return launch_window((int)n, kl, ku, (int)nrhs, AB, (int)ldab, ipiv, B, ldb, d_info, s);
    if (wide_fits(win - 1)) return launch_wide((int)n, kl, ku, (int)nrhs, AB, (int)ldab, ipiv, B, ldb, d_info, s);
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
