// gbtrf_wide.cu -- banded LU for wide bands (kl beyond the windowed kernel):
// persistent, cooperatively launched kernels, one CTA per SM (Sec. II-A step 3;
// f(N) ~ O(N*P*Q), Eq. S-N-N3).  Three variants share the step functions below:
//
//  * k_gbtrf_wide_chain (gbtrf_wide_stream.cuh), the default when a panel row
//    fits one thread: CTA 0 only factors, and the lookahead panels stream down a
//    cluster of streaming CTAs;
//  * k_gbtrf_wide_pair, when the chain's clusters cannot all be resident: CTA 0
//    factors and looks ahead, a second lookahead group runs on its cluster
//    partner;
//  * k_gbtrf_wide (described first, below), the single panel CTA, for up to four
//    rows per thread and wherever no cluster kernel fits.
//
// Columns are cut into blocks of kNB; block p is panel p.
//
//  * CTA 0 (panel CTA).  Group A (nine warps) owns the rows of the current
//    panel (thread i <-> row p*kNB + i, held in registers).  One panel step is
//    one exact argmax round and ONE barrier: every warp publishes its best
//    candidate together with that row's panel values, and the thread of row j
//    publishes row j, so every thread can apply the interchange, form its
//    multiplier and update its own row without further synchronisation.
//    After panel p group A applies panel p to block p+1, which thereby becomes
//    panel p+1.  Group B (nine more warps) has meanwhile applied panel p-1 to
//    block p+1, while group A factored panel p (a two-panel lookahead split
//    over two warp groups, so that only one lookahead pass is on the serial
//    path).  A storer warp writes every finished panel block and its pivots to
//    AB and ipiv and publishes them (panel_ready[p]); a loader warp brings
//    block b in with cp.async once its owner has handed it over
//    (block_ready[b]) and its buffer is free.
//  * CTAs 1..G (update CTAs) own the blocks b >= 3, block b on CTA
//    1 + (b-3) mod G.  A block is read into shared memory when the first panel
//    reaching it is published, receives panels p_first(b)..b-3 in order, and is
//    handed to the panel CTA (written to AB, block_ready[b]) two panels before
//    the panel CTA needs it.
//
// Every entry receives exactly the fma sequence of the unblocked elimination
// in the same order (the interchanges permute the same values, the multiplier
// is the pivot's correctly rounded reciprocal times the entry, each update is
// fma(-l, u, a) with the zero-u skip), so the factors are bit-identical to it.
// Interchanges and updates are applied up to the band's reach j + kv instead
// of the running column reach ju: beyond ju both interchanged entries and the
// row-j entry are +0.0 fill, so this changes no bit.
//
// Hand-offs between CTAs are acquire/release flags in global memory, inside
// the panel CTA mbarrier rings (a ring of kRing entries per hand-off, deeper
// than any producer can run ahead of its consumer); every wait is bounded.  A wait that gives up raises
// an error flag that every waiter checks, the kernel ends, and *d_info becomes
// -BANDLU_ERR_TIMEOUT.
#include <algorithm>
#include <climits>
#include <cstdint>
#include <cstdlib>
#include <map>
#include <mutex>
#include <tuple>

#include "bandlu_trace.h"
#include "common.cuh"
#include "rcp.cuh"
#include "sync.cuh"

namespace bandlu {
namespace {

constexpr int kNB = 4;                // panel width = column block width
// A compute group has CW warps (a template parameter: 2, 4 or 9, the fewest that
// give every row of a panel, kl + kNB of them, its own thread).  The panel CTA
// runs two groups (A: warps 0..CW-1, B: CW..2CW-1), a storer and a loader warp.
template <int CW>
struct Lay {
  static constexpr int kCT = 32 * CW;            // threads of a compute group
  static constexpr int kStoreWarp = 2 * CW;
  static constexpr int kLoadWarp = kStoreWarp + 1;
  static constexpr int kThreads = 32 * (kLoadWarp + 1);
};
constexpr int kBarA = 1, kBarB = 2;   // named barriers of the two groups
constexpr int kRing = 4;              // depth of the hand-off mbarrier rings
constexpr int kMaxActive = 2;         // blocks an update CTA holds at once
constexpr int kPanelBufs = 3;         // block buffers of the panel CTA
constexpr long long kSpinLimit = 2000000000ll;

template <int CW>
__device__ __forceinline__ void bar_group(int id) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "n"(Lay<CW>::kCT) : "memory");
}
template <int CW>
__device__ __forceinline__ void bar_compute() { bar_group<CW>(kBarA); }

__device__ __forceinline__ int ld_acquire(const int *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ int ld_relaxed(const int *p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int *p, int v) {
  asm volatile("st.release.gpu.global.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Pivot-search key of a candidate, so that the FIRST largest key is the row
// the xGBTRF comparison order picks: the running best starts at the first
// candidate and a later one replaces it only if strictly larger in modulus.
// NaN never compares larger, so it wins only as the first candidate.  Keys are
// offset by one so that 0 means "not a candidate".
__device__ __forceinline__ unsigned long long pivot_key(double a, bool first) {
  const unsigned hi = (unsigned)__double2hiint(a) & 0x7fffffffu, lo = (unsigned)__double2loint(a);
  const bool nan = hi > 0x7ff00000u || (hi == 0x7ff00000u && lo != 0u);
  const unsigned long long b = ((unsigned long long)hi << 32) | lo;
  return nan ? (first ? 0x8000000000000000ull : 1ull) : b + 1ull;
}

// First lane holding the largest key; *kmax receives that key.
__device__ __forceinline__ int warp_first_max(unsigned long long key, unsigned long long *kmax) {
  const unsigned hi = (unsigned)(key >> 32), lo = (unsigned)key;
  const unsigned mhi = __reduce_max_sync(FULL, hi);
  const unsigned mlo = __reduce_max_sync(FULL, hi == mhi ? lo : 0u);
  *kmax = ((unsigned long long)mhi << 32) | mlo;
  return __ffs(__ballot_sync(FULL, hi == mhi && lo == mlo)) - 1;
}

// Bit d set iff u[d] != 0.0.
__device__ __forceinline__ unsigned nz_mask(const double (&u)[kNB]) {
  unsigned m = 0;
#pragma unroll
  for (int d = 0; d < kNB; ++d) m |= nz(u[d]) ? (1u << d) : 0u;
  return m;
}
// One elimination update a - l*u with the zero-u skip (unz = u != 0), branch
// free: the fma is always issued and its result discarded when u is +-0 (so a
// signed zero a and an infinite l stay as the skip leaves them).
__device__ __forceinline__ double upd(double l, double u, double a, bool unz) {
  const double t = fma(-l, u, a);
  return unz ? t : a;
}

struct Geo {
  int n, kl, ku, kv;
  long long ldab;
  int npan;
  bool vec;  // AB is 16-byte aligned: blocks move as 16-byte chunks
};

// First panel whose U rows reach block b (panel p reaches column (p+1)*kNB - 1 + kv).
__device__ __forceinline__ int p_first(const Geo &g, int b) {
  const int x = b * kNB - g.kv + 1;
  return x <= 0 ? 0 : (x + kNB - 1) / kNB - 1;
}
// Last block reached by panel p.
__device__ __forceinline__ int b_last(const Geo &g, int p) {
  return min(g.npan - 1, ((p + 1) * kNB - 1 + g.kv) / kNB);
}
// Block b passes through an update CTA (which applies panels p_first(b)..b-3).
__device__ __forceinline__ bool handed_off(const Geo &g, int b) { return b >= 3 && p_first(g, b) <= b - 3; }

// Synchronisation and broadcast state.  Slots indexed [2] alternate with the
// barrier count: a slot is rewritten only two barriers after it was published,
// when every reader has passed the barrier in between.
// Broadcast slots of one compute group's lookahead steps.
struct Bcast {
  double bu[2][kNB];   // pivot row in the block's columns
  double br0[2][kNB];  // row j in the block's columns
  unsigned bum[2];     // nonzero mask of bu
};

template <int CW, int RPT>
struct WideShared {
  static constexpr int kCW = CW;
  unsigned long long key[2][RPT * kCW];
  double piv[2][RPT * kCW][kNB];  // each warp's best candidate row, panel columns
  int idx[2][RPT * kCW];
  double row0[2][kNB];            // row j before the interchange, panel columns
  unsigned pivm[2][RPT * kCW];    // nonzero masks of piv
  double prc[2][RPT * kCW];       // correctly rounded reciprocal of each partial's candidate
  int pspec[2][RPT * kCW];        // ... not formed (zero, subnormal, huge, inf, nan)
  Bcast bc[2];                    // group A, group B
  int pk[2][kNB];                 // pivot offsets of a panel, by panel parity
  int zp[2][kNB];                 // exact zero pivot
  int pvr[kRing][kNB];            // pivot offsets for the storer, by panel
  // hand-off rings: entry i of a ring serves events i, i+kRing, ... (parity = which)
  unsigned long long mb_done[kRing];    // A -> storer: panel p finished          (p)
  unsigned long long mb_stored[kRing];  // storer -> loader: block p written out  (p)
  unsigned long long mb_go[kRing];      // A -> B: panel b-2 finished            (b-2)
  unsigned long long mb_loaded[kRing];  // loader -> B: block b in shared memory (b-2)
  unsigned long long mb_bdone[kRing];   // B -> A: panel b-2 applied to block b  (b-2)
  int ok[2];
  int info;
};

// ---- bounded waits ------------------------------------------------------------

// Polls `ready` until it returns true; gives up (false) when *err is raised or
// the cycle budget runs out (then raises *err itself).
template <class F>
__device__ __forceinline__ bool bounded_poll(F ready, int *err) {
  if (ready()) return true;
  const long long t0 = clock64();
  for (unsigned it = 1;; ++it) {
    if (ready()) return true;
    if ((it & 15u) == 0u) {
      if (ld_relaxed(err) != 0) return false;
      if (clock64() - t0 > kSpinLimit) {
        atomicExch(err, 1);
        return false;
      }
    }
  }
}

// All threads of a compute group (tid = index in the group): its thread 0
// waits, the outcome is shared.
template <int CW, int RPT, class F>
__device__ bool group_wait(F ready, int *err, WideShared<CW, RPT> &sh, int tid, int grp) {
  if (tid == 0) sh.ok[grp] = bounded_poll(ready, err) ? 1 : 0;
  bar_group<CW>(grp == 0 ? kBarA : kBarB);
  const bool ok = sh.ok[grp] != 0;
  bar_group<CW>(grp == 0 ? kBarA : kBarB);
  return ok;
}
template <int CW, int RPT, class F>
__device__ bool compute_wait(F ready, int *err, WideShared<CW, RPT> &sh) {
  return group_wait<CW, RPT>(ready, err, sh, threadIdx.x, 0);
}

// I/O warp: lane 0 waits, the outcome is warp-uniform.
template <class F>
__device__ bool io_wait(F ready, int *err) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = bounded_poll(ready, err) ? 1 : 0;
  ok = __shfl_sync(FULL, ok, 0);
  __syncwarp();
  return ok != 0;
}

// ---- block transfers ------------------------------------------------------------
// A block is kNB columns of AB (kNB * ldab doubles, the last block fewer).
// first: the block's first read, so its fill rows 0..kl-1 are cleared (the
// elimination clears every fill row before it starts).

__device__ void load_block(const Geo &g, const double *AB, double *blk, int b, bool first, int t, int nt) {
  const int c0 = b * kNB, nc = min(kNB, g.n - c0);
  const int tot = nc * (int)g.ldab;
  const double *src = AB + (long long)c0 * g.ldab;
  if (first || !g.vec) {
    for (int e = t; e < tot; e += nt) {
      const int r = e % (int)g.ldab;
      blk[e] = (first && r < g.kl) ? 0.0 : __ldcg(src + e);
    }
  } else {
    for (int e = 2 * t; e + 1 < tot; e += 2 * nt)
      reinterpret_cast<double2 *>(blk)[e >> 1] = __ldcg(reinterpret_cast<const double2 *>(src) + (e >> 1));
    if ((tot & 1) && t == 0) blk[tot - 1] = __ldcg(src + tot - 1);
  }
}

__device__ void store_block(const Geo &g, double *AB, const double *blk, int b, int t, int nt) {
  const int c0 = b * kNB, nc = min(kNB, g.n - c0);
  const int tot = nc * (int)g.ldab;
  double *dst = AB + (long long)c0 * g.ldab;
  if (!g.vec) {
    for (int e = t; e < tot; e += nt) dst[e] = blk[e];
  } else {
    for (int e = 2 * t; e + 1 < tot; e += 2 * nt)
      reinterpret_cast<double2 *>(dst)[e >> 1] = reinterpret_cast<const double2 *>(blk)[e >> 1];
    if ((tot & 1) && t == 0) dst[tot - 1] = blk[tot - 1];
  }
}

// Loader: one bulk (TMA) copy of a handed-off block of kNB full columns
// (kNB * ldab * 8 bytes, a multiple of 16 with AB 16-byte aligned); it
// completes the phase of *mbar once the bytes have landed.  The block was
// written through ordinary stores by another CTA and acquired through its flag,
// so the generic-to-async proxy fence comes first.
__device__ void bulk_prefetch_block(const Geo &g, const double *AB, double *blk, int b, unsigned long long *mbar) {
  const unsigned bytes = (unsigned)(kNB * g.ldab * sizeof(double));
  const double *src = AB + (long long)b * kNB * g.ldab;
  asm volatile("fence.proxy.async.global;" ::: "memory");
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(mbar)), "r"(bytes)
               : "memory");
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_addr(blk)),
               "l"(src), "r"(bytes), "r"(smem_addr(mbar))
               : "memory");
}

// I/O warp: copy of a handed-off block in 16-byte cp.async chunks (AB aligned).
__device__ void io_prefetch_block(const Geo &g, const double *AB, double *blk, int b) {
  const int lane = threadIdx.x & 31;
  const int c0 = b * kNB, nc = min(kNB, g.n - c0);
  const int tot = nc * (int)g.ldab;
  const double *src = AB + (long long)c0 * g.ldab;
  for (int e = 2 * lane; e + 1 < tot; e += 64) {
    const unsigned d = smem_addr(blk + e);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src + e) : "memory");
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  if ((tot & 1) && lane == 0) blk[tot - 1] = __ldcg(src + tot - 1);
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

// ---- one panel applied to a later block -----------------------------------------
// Compute threads; thread i <-> row q*kNB + i (the rows of panel q's steps).
// lr[r][k]: multiplier of the thread's row r at step k (0 if none).  The slot
// parity `bpar` advances at each barrier.
template <int CW, int RPT>
__device__ void apply_panel(const Geo &g, double *blk, int b, int q, const double (&lr)[RPT][kNB], const int *pk,
                            const int *zp, Bcast &bc, int tid, int bar, int &bpar) {
  constexpr int kCT = Lay<CW>::kCT;
  const int c0q = q * kNB, ncq = min(kNB, g.n - c0q);
  const int c0b = b * kNB, ncb = min(kNB, g.n - c0b);
  const int ldab = (int)g.ldab;
  double w[RPT][kNB];
#pragma unroll
  for (int r = 0; r < RPT; ++r) {
    const int i = tid + r * kCT, row = c0q + i;
#pragma unroll
    for (int d = 0; d < kNB; ++d) {
      const int pos = g.kv + row - (c0b + d);
      const bool ok = i < g.kl + kNB && row < g.n && d < ncb && pos >= 0;
      w[r][d] = ok ? blk[d * ldab + pos] : 0.0;
    }
  }
#pragma unroll
  for (int k = 0; k < kNB; ++k) {
    if (k >= ncq) break;
    if (zp[k]) continue;  // uniform
    const int j = c0q + k, km = min(g.kl, g.n - 1 - j), p = pk[k];
    const int s = bpar;
    bpar ^= 1;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int i = tid + r * kCT;
      if (i == k + p) {
#pragma unroll
        for (int d = 0; d < kNB; ++d) bc.bu[s][d] = w[r][d];
        bc.bum[s] = nz_mask(w[r]);
      }
      if (i == k) {
#pragma unroll
        for (int d = 0; d < kNB; ++d) bc.br0[s][d] = w[r][d];
      }
    }
    bar_group<CW>(bar);
    double u[kNB];
#pragma unroll
    for (int d = 0; d < kNB; ++d) u[d] = bc.bu[s][d];
    const unsigned um = bc.bum[s];
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int i = tid + r * kCT;
      if (i == k) {
#pragma unroll
        for (int d = 0; d < kNB; ++d) w[r][d] = u[d];
      } else if (p != 0 && i == k + p) {
#pragma unroll
        for (int d = 0; d < kNB; ++d) w[r][d] = bc.br0[s][d];
      }
      if (i > k && i <= k + km) {
        const double l = lr[r][k];
#pragma unroll
        for (int d = 0; d < kNB; ++d) w[r][d] = upd(l, u[d], w[r][d], (um >> d) & 1u);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < RPT; ++r) {
    const int i = tid + r * kCT, row = c0q + i;
#pragma unroll
    for (int d = 0; d < kNB; ++d) {
      const int pos = g.kv + row - (c0b + d);
      if (i < g.kl + kNB && row < g.n && d < ncb && pos >= 0) blk[d * ldab + pos] = w[r][d];
    }
  }
}

// ---- panel factorisation (panel CTA compute threads) -----------------------------
// Factors block p in place; records the pivot offsets and zero flags in
// sh.pk/sh.zp[p & 1] and the multipliers in s_l (s_l[k*kl + t-1] = l_{j+t, j},
// j = p*kNB + k).
template <int CW, int RPT>
__device__ void factor_panel(const Geo &g, double *blk, int p, double *s_l, WideShared<CW, RPT> &sh, int &bpar,
                             int &info) {
  constexpr int kCT = Lay<CW>::kCT, kCW = CW;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c0 = p * kNB, nc = min(kNB, g.n - c0);
  const int ldab = (int)g.ldab;
  const int pp = p & 1;
  double v[RPT][kNB];
#pragma unroll
  for (int r = 0; r < RPT; ++r) {
    const int i = tid + r * kCT, row = c0 + i;
#pragma unroll
    for (int k = 0; k < kNB; ++k) {
      const bool ok = i < g.kl + kNB && row < g.n && k < nc && i - k <= g.kl;
      v[r][k] = ok ? blk[k * ldab + g.kv + i - k] : 0.0;
    }
  }
#pragma unroll
  for (int k = 0; k < kNB; ++k) {
    if (k >= nc) break;
    const int j = c0 + k, km = min(g.kl, g.n - 1 - j);
    const int s = bpar;
    bpar ^= 1;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
      const int i = tid + r * kCT, t = i - k;
      // every thread forms the reciprocal of its own candidate while the argmax runs
      bool myspec;
      const double myr = rcp_rn_fast(v[r][k], &myspec);
      const unsigned long long key = (t >= 0 && t <= km) ? pivot_key(v[r][k], t == 0) : 0ull;
      unsigned long long kmax;
      const int wl = warp_first_max(key, &kmax);
      if (lane == wl) {
        sh.key[s][r * kCW + warp] = kmax;
        sh.idx[s][r * kCW + warp] = i;
#pragma unroll
        for (int d = 0; d < kNB; ++d) sh.piv[s][r * kCW + warp][d] = v[r][d];
        sh.pivm[s][r * kCW + warp] = nz_mask(v[r]);
        sh.prc[s][r * kCW + warp] = myr;
        sh.pspec[s][r * kCW + warp] = myspec ? 1 : 0;
      }
      if (i == k) {
#pragma unroll
        for (int d = 0; d < kNB; ++d) sh.row0[s][d] = v[r][d];
      }
    }
    bar_compute<CW>();
    // the first largest key over the partials, which are in row order: one lane per
    // partial and a warp argmax (lowest lane on ties), instead of a serial scan
    int wb = 0;
    if constexpr (RPT * kCW <= 32) {
      const unsigned long long kx = lane < RPT * kCW ? sh.key[s][lane] : 0ull;
      unsigned long long kbest;
      wb = warp_first_max(kx, &kbest);
    } else {
      unsigned long long best = sh.key[s][0];
#pragma unroll
      for (int x = 1; x < RPT * kCW; ++x) {
        const unsigned long long kx = sh.key[s][x];
        if (kx > best) {
          best = kx;
          wb = x;
        }
      }
    }
    const int p_off = sh.idx[s][wb] - k;
    double u[kNB];
#pragma unroll
    for (int d = 0; d < kNB; ++d) u[d] = sh.piv[s][wb][d];
    const unsigned um = sh.pivm[s][wb];
    const bool zero = ((um >> k) & 1u) == 0u;
    if (tid == 0) {
      sh.pk[pp][k] = p_off;
      sh.zp[pp][k] = zero ? 1 : 0;
      if (zero && info == 0) info = j + 1;
    }
    if (!zero) {
      double rc = sh.prc[s][wb];
      if (sh.pspec[s][wb]) rc = rcp_division(u[k]);  // uniform
#pragma unroll
      for (int r = 0; r < RPT; ++r) {
        const int i = tid + r * kCT;
        if (i == k) {
#pragma unroll
          for (int d = 0; d < kNB; ++d)
            if (d >= k) v[r][d] = u[d];
        } else if (p_off != 0 && i == k + p_off) {
#pragma unroll
          for (int d = 0; d < kNB; ++d)
            if (d >= k) v[r][d] = sh.row0[s][d];
        }
        if (i > k && i <= k + km) {
          const double l = v[r][k] * rc;
          v[r][k] = l;
#pragma unroll
          for (int d = 0; d < kNB; ++d)
            if (d > k) v[r][d] = upd(l, u[d], v[r][d], (um >> d) & 1u);
        }
      }
    }
  }
#pragma unroll
  for (int r = 0; r < RPT; ++r) {
    const int i = tid + r * kCT, row = c0 + i;
#pragma unroll
    for (int k = 0; k < kNB; ++k) {
      if (i < g.kl + kNB && row < g.n && k < nc && i - k <= g.kl) blk[k * ldab + g.kv + i - k] = v[r][k];
      const int t = i - k;
      if (k < nc && t >= 1 && t <= min(g.kl, g.n - 1 - (c0 + k))) s_l[k * g.kl + t - 1] = v[r][k];
    }
  }
}

// Multipliers of panel q for the rows of a compute group's threads (tid in the
// group): lr[r][k] = l_{j+t, j}, j = q*kNB + k, t = tid + r*kCT - k.
template <int CW, int RPT>
__device__ __forceinline__ void panel_multipliers(const Geo &g, const double *ql, int q, int tid,
                                                  double (&lr)[RPT][kNB]) {
  constexpr int kCT = Lay<CW>::kCT;
  const int c0q = q * kNB;
#pragma unroll
  for (int r = 0; r < RPT; ++r) {
    const int i = tid + r * kCT;
#pragma unroll
    for (int k = 0; k < kNB; ++k) {
      const int t = i - k;
      lr[r][k] = (c0q + k < g.n && t >= 1 && t <= min(g.kl, g.n - 1 - (c0q + k))) ? ql[k * g.kl + t - 1] : 0.0;
    }
  }
}

template <int CW, int RPT>
__global__ void __launch_bounds__(Lay<CW>::kThreads, 1)
    k_gbtrf_wide(Geo g, double *__restrict__ AB, int *__restrict__ ipiv, int *__restrict__ d_info,
                 int *__restrict__ flags) {
  constexpr int kCT = Lay<CW>::kCT, kCW = CW, kStoreWarp = Lay<CW>::kStoreWarp;
  extern __shared__ __align__(16) double smem[];
  __shared__ WideShared<CW, RPT> sh;
  int *err = flags;
  int *panel_ready = flags + 2;
  int *block_ready = flags + 2 + g.npan;
  const long long bsz = (long long)kNB * g.ldab;
  double *blocks = smem;                              // kPanelBufs (panel CTA) / kMaxActive blocks
  double *s_lbase = smem + (size_t)kPanelBufs * bsz;  // 2 panels of kNB * kl multipliers
  const int tid = threadIdx.x, warp = tid >> 5;
  auto buf = [&](int b) { return blocks + (long long)(b % kPanelBufs) * bsz; };
  auto mults = [&](int q) { return s_lbase + (size_t)(q & 1) * kNB * g.kl; };
  auto ring_par = [](int e) { return (unsigned)(e / kRing) & 1u; };

  if (blockIdx.x == 0 && tid == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&sh.mb_done[i], 1);
      mbar_init(&sh.mb_stored[i], 1);
      mbar_init(&sh.mb_go[i], 1);
      mbar_init(&sh.mb_loaded[i], 1);
      mbar_init(&sh.mb_bdone[i], 1);
    }
    sh.info = 0;
  }
  __syncthreads();

  if (blockIdx.x == 0) {
    if (warp < kCW) {
      // ---------------- panel CTA, group A: factorisation and lookahead of panel p ----------------
      int info = 0, bpar = 0;
      load_block(g, AB, buf(0), 0, true, tid, kCT);
      if (g.npan > 1) load_block(g, AB, buf(1), 1, true, tid, kCT);
      bar_compute<CW>();
      for (int p = 0; p < g.npan; ++p) {
        factor_panel<CW, RPT>(g, buf(p), p, mults(p), sh, bpar, info);
        if (tid == 0) {
          sh.info = info;
#pragma unroll
          for (int k = 0; k < kNB; ++k) sh.pvr[p % kRing][k] = sh.pk[p & 1][k];
        }
        bar_compute<CW>();
        if (tid == 0) {
          mbar_arrive(&sh.mb_done[p % kRing]);
          if (p + 2 < g.npan) mbar_arrive(&sh.mb_go[p % kRing]);  // B may apply panel p to block p+2
        }
        if (p + 1 < g.npan) {
          const int b = p + 1;
          // block b holds panels <= b-2 (update CTAs and group B)
          if (b >= 2) {
            unsigned long long *mb = &sh.mb_bdone[(b - 2) % kRing];
            const unsigned par = ring_par(b - 2);
            if (!compute_wait<CW, RPT>([&] { return mbar_try_wait(mb, par); }, err, sh)) break;
          }
          if (p >= p_first(g, b)) {  // uniform
            double lr[RPT][kNB];
            panel_multipliers<CW, RPT>(g, mults(p), p, tid, lr);
            apply_panel<CW, RPT>(g, buf(b), b, p, lr, sh.pk[p & 1], sh.zp[p & 1], sh.bc[0], tid, kBarA, bpar);
            bar_compute<CW>();
          }
        }
      }
    } else if (warp < kStoreWarp) {
      // ---------------- panel CTA, group B: panel b-2 applied to block b ----------------
      const int tidb = tid - kCT;
      int bpar = 0;
      for (int b = 2; b < g.npan; ++b) {
        unsigned long long *mg = &sh.mb_go[(b - 2) % kRing];
        unsigned long long *ml = &sh.mb_loaded[(b - 2) % kRing];
        const unsigned par = ring_par(b - 2);
        if (!group_wait<CW, RPT>([&] { return mbar_try_wait(mg, par); }, err, sh, tidb, 1)) break;
        if (!group_wait<CW, RPT>([&] { return mbar_try_wait(ml, par); }, err, sh, tidb, 1)) break;
        const int q = b - 2;
        if (q >= p_first(g, b)) {  // uniform
          double lr[RPT][kNB];
          panel_multipliers<CW, RPT>(g, mults(q), q, tidb, lr);
          apply_panel<CW, RPT>(g, buf(b), b, q, lr, sh.pk[q & 1], sh.zp[q & 1], sh.bc[1], tidb, kBarB, bpar);
        }
        bar_group<CW>(kBarB);
        if (tidb == 0) mbar_arrive(&sh.mb_bdone[(b - 2) % kRing]);
      }
    } else if (warp == kStoreWarp) {
      // ---------------- panel CTA, storer: finished panels to AB, published ----------------
      const int lane = tid & 31;
      for (int p = 0; p < g.npan; ++p) {
        unsigned long long *mb = &sh.mb_done[p % kRing];
        const unsigned par = ring_par(p);
        if (!io_wait([&] { return mbar_try_wait(mb, par); }, err)) break;
        const int c0 = p * kNB, nc = min(kNB, g.n - c0);
        const double *src = buf(p);
        double *dst = AB + (long long)c0 * g.ldab;
        const int ld = (int)g.ldab;
        // what the update CTAs read first: the diagonal and the multipliers (rows
        // kv..kv+kl of the panel's columns) and the pivots; then the publication
        for (int k = 0; k < nc; ++k)
          for (int rr = g.kv + lane; rr <= g.kv + g.kl; rr += 32) dst[k * ld + rr] = src[k * ld + rr];
        if (lane < nc) ipiv[c0 + lane] = c0 + lane + sh.pvr[p % kRing][lane] + 1;
        __threadfence();
        __syncwarp();
        if (lane == 0) st_release(panel_ready + p, 1);
        // then the whole block (the published rows again, unchanged)
        store_block(g, AB, src, p, lane, 32);
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.mb_stored[p % kRing]);  // its buffer may take block p+3
      }
      // info is final once the last panel is done; the status reflects every CTA's waits
      if (lane == 0) *d_info = ld_acquire(err) ? -BANDLU_ERR_TIMEOUT : sh.info;
    } else {
      // ---------------- panel CTA, loader: blocks b >= 2 into shared memory ----------------
      const int lane = tid & 31;
      for (int b = 2; b < g.npan; ++b) {
        if (b >= 3) {  // the buffer held block b-3
          unsigned long long *mb = &sh.mb_stored[(b - 3) % kRing];
          const unsigned par = ring_par(b - 3);
          if (!io_wait([&] { return mbar_try_wait(mb, par); }, err)) break;
        }
        double *dst = buf(b);
        unsigned long long *ml = &sh.mb_loaded[(b - 2) % kRing];
        if (handed_off(g, b)) {
          const int *f = block_ready + b;
          if (!io_wait([&] { return ld_acquire(f) != 0; }, err)) break;
          if (g.vec && (b + 1) * kNB <= g.n) {
            if (lane == 0) bulk_prefetch_block(g, AB, dst, b, ml);  // completes the phase itself
            __syncwarp();
            continue;
          }
          if (g.vec) {
            io_prefetch_block(g, AB, dst, b);
          } else {
            load_block(g, AB, dst, b, false, lane, 32);
          }
        } else {
          load_block(g, AB, dst, b, true, lane, 32);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(ml);
      }
    }
  } else {
    // ---------------- update CTAs ----------------
    if (warp >= kCW) return;
    const int G = gridDim.x - 1, u = blockIdx.x - 1;
    int bpar = 0;
    for (int p = 0; p + 3 < g.npan; ++p) {
      // owned blocks that panel p updates here: b in [p+3, b_last(p)], b = 3 + u (mod G)
      const int lo = p + 3, hi = b_last(g, p);
      const int b0 = lo + ((u - (lo - 3)) % G + G) % G;
      if (b0 > hi) continue;
      const int *f = panel_ready + p;
      if (!compute_wait<CW, RPT>([&] { return ld_acquire(f) != 0; }, err, sh)) break;
      const int c0q = p * kNB, ncq = min(kNB, g.n - c0q);
      if (tid < kNB) {
        const int k = tid;
        sh.pk[0][k] = k < ncq ? __ldcg(ipiv + c0q + k) - 1 - (c0q + k) : 0;
        sh.zp[0][k] = k < ncq ? (nz(__ldcg(AB + (long long)(c0q + k) * g.ldab + g.kv)) ? 0 : 1) : 1;
      }
      double lr[RPT][kNB];
#pragma unroll
      for (int r = 0; r < RPT; ++r) {
        const int i = tid + r * kCT;
#pragma unroll
        for (int k = 0; k < kNB; ++k) {
          const int t = i - k;
          lr[r][k] = (k < ncq && t >= 1 && t <= min(g.kl, g.n - 1 - (c0q + k)))
                         ? __ldcg(AB + (long long)(c0q + k) * g.ldab + g.kv + t)
                         : 0.0;
        }
      }
      bar_compute<CW>();
      for (int b = b0; b <= hi; b += G) {
        double *blk = blocks + (long long)(((b - 3) / G) % kMaxActive) * bsz;
        if (p == p_first(g, b)) {
          load_block(g, AB, blk, b, true, tid, kCT);
          bar_compute<CW>();
        }
        apply_panel<CW, RPT>(g, blk, b, p, lr, sh.pk[0], sh.zp[0], sh.bc[0], tid, kBarA, bpar);
        bar_compute<CW>();
        if (p == b - 3) {
          store_block(g, AB, blk, b, tid, kCT);
          __threadfence();
          bar_compute<CW>();
          if (tid == 0) st_release(block_ready + b, 1);
        }
      }
    }
  }
}

// ==== the cluster-pair variant ==================================================
//
// GB300's FP64 unit of an SM sub-partition accepts one warp instruction about
// every 64-76 clocks, whatever the number of active lanes, so the panel CTA's
// pace is set by the FP64 instructions queued on its four sub-partitions: group
// A's factor steps and lookahead (26 per row per panel) and group B's lookahead
// (16 per row per panel), with B's multiply-adds queued in front of A's
// critical ones.  Here group B runs on its own SM, CTA 1 of a two-CTA cluster:
//
//  * CTA 0 (A): group A factors panel p and applies it to block p+1, as above,
//    keeping the last kRB panels' multipliers and pivots in a ring in shared
//    memory.  A storer warp writes finished panels to AB, publishes them, and
//    tells CTA 1 that panel p's multipliers are ready; CTA 1 reads them from the
//    ring through distributed shared memory and returns the entry when done.
//  * CTA 1 (B): group B applies panel q to block q+2 and sends that block into
//    CTA 0's shared memory (where it arrives as block p+1 of panel p = q+1)
//    (and, with kHand = 4, then applies panel q to block q+3).  A loader warp
//    brings each block in from AB (a bulk copy once its update CTA hands it
//    over, else a fresh load).
//  * CTAs 2.. (update CTAs) own the blocks b >= kHand round-robin, apply panels
//    p_first(b)..b-kHand and hand the block over (block_ready[b]).
//
// Every element still receives the unblocked elimination's fma sequence in the
// same order (panels are applied to a block in increasing order by whichever CTA
// holds it), so the factors are bit-identical.  Cross-CTA data moves with plain
// loads and stores through distributed shared memory; after its stores each warp
// (or the one signalling thread, after the group's barrier) arrives with release
// semantics at cluster scope on the receiving CTA's mbarrier, and the receivers
// wait on it with acquire at cluster scope.  Group A's own path has no remote
// operation.  Nothing is asynchronous between the two CTAs, so when both have
// passed the final cluster barrier no transfer is in flight.
// Every wait is bounded, as in the single-CTA panel kernel.

constexpr int kRB = 4;      // multiplier ring entries (panels) on CTA 0
constexpr int kBBufs = 4;   // block buffers on CTA 1
// Update CTAs apply panels p_first(b)..b-kHand to block b and hand it over; CTA 1
// applies panels b-kHand+1..b-2 (one per panel period for each value of kHand - 2).
constexpr int kHand = 3;

template <int CW>
struct PairShared {
  WideShared<CW, 1> w;
  unsigned long long mb_mult[kRB];     // CTA 1: panel q factored, its multipliers in CTA 0's ring (1 arrival, storer)
  unsigned long long mb_credit[kRB];   // CTA 0: CTA 1 has read ring entry q % kRB (1 arrival)
  unsigned long long mb_blk[kRing];    // CTA 0: block b arrived in buf(b), event b-2 (one arrival per warp of B)
  unsigned long long mb_afree[kRing];  // CTA 1: CTA 0's buffer of panel p stored, event p (1 arrival, storer)
  unsigned long long mb_bload[kBBufs]; // CTA 1: block b in its buffer, event b-2 (loader)
  unsigned long long mb_bsent[kBBufs]; // CTA 1: block b sent, its buffer free, event b-2 (group B)
  int rpk[kRB][kNB];                   // CTA 0: pivot offsets of the ring's panels (read by CTA 1)
  int rzp[kRB][kNB];                   // CTA 0: exact-zero-pivot flags of the ring's panels
};

__device__ __forceinline__ unsigned cl_map(const void *p, unsigned rank) {
  unsigned r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
  return r;
}
// Generic address of the same shared-memory object in CTA `rank` of the cluster;
// ordinary loads and stores through it reach that CTA's shared memory.
template <class T>
__device__ __forceinline__ T *cl_generic(T *p, unsigned rank) {
  unsigned long long r;
  asm volatile("mapa.u64 %0, %1, %2;" : "=l"(r) : "l"(reinterpret_cast<unsigned long long>(p)), "r"(rank));
  return reinterpret_cast<T *>(r);
}
__device__ __forceinline__ void cl_st2(unsigned raddr, double a, double b) {
  asm volatile("st.shared::cluster.v2.f64 [%0], {%1, %2};" ::"r"(raddr), "d"(a), "d"(b) : "memory");
}
__device__ __forceinline__ void cl_st1(unsigned raddr, double a) {
  asm volatile("st.shared::cluster.f64 [%0], %1;" ::"r"(raddr), "d"(a) : "memory");
}
// One arrival on an mbarrier of CTA `rank`, ordering this thread's earlier
// memory operations before it at cluster scope.
__device__ __forceinline__ void cl_arrive(const unsigned long long *bar, unsigned rank) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cl_map(bar, rank)) : "memory");
}
__device__ __forceinline__ bool cl_try_wait(unsigned long long *bar, unsigned parity) {
  unsigned ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void cluster_barrier() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ unsigned ring_parity(int e, int R) { return (unsigned)(e / R) & 1u; }

// Blocks b >= kHand pass through an update CTA, which applies panels p_first(b)..b-kHand.
__device__ __forceinline__ bool handed_off_pair(const Geo &g, int b) {
  return b >= kHand && p_first(g, b) <= b - kHand;
}

template <int CW>
__global__ void __launch_bounds__(32 * (CW + 1), 1)
    k_gbtrf_wide_pair(Geo g0, double *__restrict__ AB, int *__restrict__ ipiv, int *__restrict__ d_info,
                      int *__restrict__ flags, const int *__restrict__ d_kl, const int *__restrict__ d_ku) {
  constexpr int kCT = Lay<CW>::kCT, kCW = CW;
  Geo g = g0;
  if (d_kl != nullptr) {
    // enqueued by the device-side dispatch before the bandwidths were known: the
    // decision (flags[1], set by the kernel before this one) and (kl, ku) are read
    // here, by every CTA alike, so either all of them work or all leave now
    if (*(volatile const int *)(flags + 1) == 0) return;
    g.kl = *d_kl;
    g.ku = *d_ku;
    g.kv = g.kl + g.ku;
  }
  extern __shared__ __align__(16) double smem[];
  __shared__ PairShared<CW> ps;
  WideShared<CW, 1> &sh = ps.w;
  int *err = flags;
  int *panel_ready = flags + 2;
  int *block_ready = flags + 2 + g.npan;
  const long long bsz = (long long)kNB * g.ldab;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // CTA 0: kPanelBufs block buffers and a ring of kRB panels of multipliers; CTA 1: kBBufs
  // block buffers; update CTAs: kMaxActive block buffers
  double *blocks = smem;
  double *s_lbase = smem + (size_t)kPanelBufs * bsz;
  auto buf = [&](int b) { return blocks + (long long)(b % kPanelBufs) * bsz; };
  auto bbuf = [&](int b) { return blocks + (long long)((b - 2) % kBBufs) * bsz; };
  auto mults = [&](int q) { return s_lbase + (size_t)(q % kRB) * kNB * g.kl; };

  if (tid == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&sh.mb_done[i], 1);
      mbar_init(&sh.mb_stored[i], 1);
      mbar_init(&ps.mb_blk[i], kCW);
      mbar_init(&ps.mb_afree[i], 1);
    }
    for (int i = 0; i < kRB; ++i) {
      mbar_init(&ps.mb_mult[i], 1);
      mbar_init(&ps.mb_credit[i], 1);
    }
    for (int i = 0; i < kBBufs; ++i) {
      mbar_init(&ps.mb_bload[i], 1);
      mbar_init(&ps.mb_bsent[i], 1);
    }
    sh.info = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  cluster_barrier();  // every CTA's barriers initialised before any remote arrival

  // bounded waits (all threads of a compute group, or one warp)
  auto grp_wait_cl = [&](unsigned long long *bar, unsigned par, int bar_id) -> bool {
    if (tid == 0) sh.ok[0] = bounded_poll([&] { return cl_try_wait(bar, par); }, err) ? 1 : 0;
    bar_group<CW>(bar_id);
    const bool ok = sh.ok[0] != 0;
    bar_group<CW>(bar_id);
    return ok;
  };
  auto grp_wait_local = [&](unsigned long long *bar, unsigned par, int bar_id) -> bool {
    if (tid == 0) sh.ok[0] = bounded_poll([&] { return mbar_try_wait(bar, par); }, err) ? 1 : 0;
    bar_group<CW>(bar_id);
    const bool ok = sh.ok[0] != 0;
    bar_group<CW>(bar_id);
    return ok;
  };

  if (blockIdx.x == 0) {
    if (warp < kCW) {
      // ---------------- CTA 0, group A: factorisation of panel p, lookahead to block p+1 ----------------
      int info = 0, bpar = 0;
      load_block(g, AB, buf(0), 0, true, tid, kCT);
      if (g.npan > 1) load_block(g, AB, buf(1), 1, true, tid, kCT);
      bar_compute<CW>();
      for (int p = 0; p < g.npan; ++p) {
        // ring entry p % kRB last held panel p - kRB, which CTA 1 reads: wait until it has.
        // Only a write-after-read order is needed: CTA 1's loads of the entry are performed
        // before its arrival (they precede a barrier and a release), and this CTA writes the
        // entry only after observing that arrival, so a CTA-scope poll suffices here.
        if (p >= kRB && p - kRB + 2 < g.npan &&
            !grp_wait_local(&ps.mb_credit[p % kRB], ring_parity(p - kRB, kRB), kBarA))
          break;
        factor_panel<CW, 1>(g, buf(p), p, mults(p), sh, bpar, info);
        if (tid == 0) {
          sh.info = info;
#pragma unroll
          for (int k = 0; k < kNB; ++k) {
            sh.pvr[p % kRing][k] = sh.pk[p & 1][k];
            ps.rpk[p % kRB][k] = sh.pk[p & 1][k];
            ps.rzp[p % kRB][k] = sh.zp[p & 1][k];
          }
        }
        bar_compute<CW>();
        if (tid == 0) mbar_arrive(&sh.mb_done[p % kRing]);  // the storer (which also tells CTA 1)
        double lr[1][kNB];
        panel_multipliers<CW, 1>(g, mults(p), p, tid, lr);
        if (p + 1 < g.npan) {
          const int b = p + 1;
          if (b >= 2 && !grp_wait_cl(&ps.mb_blk[(b - 2) % kRing], ring_parity(b - 2, kRing), kBarA)) break;
          if (p >= p_first(g, b)) {  // uniform
            apply_panel<CW, 1>(g, buf(b), b, p, lr, sh.pk[p & 1], sh.zp[p & 1], sh.bc[0], tid, kBarA, bpar);
            bar_compute<CW>();
          }
        }
      }
    } else if (warp == kCW) {
      // ---------------- CTA 0, storer: finished panels to AB, published ----------------
      for (int p = 0; p < g.npan; ++p) {
        unsigned long long *mb = &sh.mb_done[p % kRing];
        if (!io_wait([&] { return mbar_try_wait(mb, ring_parity(p, kRing)); }, err)) break;
        // CTA 1 applies panel p to blocks p+2 and p+3: its multipliers and pivots are
        // in the ring (ordered before group A's arrival on mb_done, which this warp acquired)
        if (p + 2 < g.npan && lane == 0) cl_arrive(&ps.mb_mult[p % kRB], 1);
        const int c0 = p * kNB, nc = min(kNB, g.n - c0);
        const double *src = buf(p);
        double *dst = AB + (long long)c0 * g.ldab;
        const int ld = (int)g.ldab;
        for (int k = 0; k < nc; ++k)
          for (int rr = g.kv + lane; rr <= g.kv + g.kl; rr += 32) dst[k * ld + rr] = src[k * ld + rr];
        if (lane < nc) ipiv[c0 + lane] = c0 + lane + sh.pvr[p % kRing][lane] + 1;
        __threadfence();
        __syncwarp();
        if (lane == 0) st_release(panel_ready + p, 1);
        store_block(g, AB, src, p, lane, 32);
        __syncwarp();
        // this buffer takes block p+3 next, which CTA 1 sends
        if (p + 3 < g.npan && lane == 0) cl_arrive(&ps.mb_afree[p % kRing], 1);
      }
      if (lane == 0) *d_info = ld_acquire(err) ? -BANDLU_ERR_TIMEOUT : sh.info;
    }
  } else if (blockIdx.x == 1) {
    if (warp < kCW) {
      // ---------------- CTA 1, group B: panel q to blocks q+2 (sent to CTA 0) and q+3 ----------------
      int bpar = 0;
      bool ok = true;
      for (int q = 0; ok && q + 2 < g.npan; ++q) {
        if (!grp_wait_cl(&ps.mb_mult[q % kRB], ring_parity(q, kRB), kBarB)) break;
        // panel q's multipliers and pivots, read from CTA 0's ring
        double lr[1][kNB];
        panel_multipliers<CW, 1>(g, cl_generic(mults(q), 0), q, tid, lr);
        int pk[kNB], zp[kNB];
        const int *rpk = cl_generic(&ps.rpk[q % kRB][0], 0), *rzp = cl_generic(&ps.rzp[q % kRB][0], 0);
#pragma unroll
        for (int k = 0; k < kNB; ++k) {
          pk[k] = rpk[k];
          zp[k] = rzp[k];
        }
        bar_group<CW>(kBarB);
        if (tid == 0) cl_arrive(&ps.mb_credit[q % kRB], 0);  // ring entry read: CTA 0 may refill it
        for (int which = 0; which <= kHand - 3; ++which) {
          const int b = q + 2 + which;
          if (b >= g.npan) break;
          // block b's first use here (panel b-kHand+1, or panel 0): wait for the loader
          if (q == max(0, b - kHand + 1)) {
            if (!grp_wait_local(&ps.mb_bload[(b - 2) % kBBufs], ring_parity(b - 2, kBBufs), kBarB)) {
              ok = false;
              break;
            }
          }
          if (q >= p_first(g, b)) {  // uniform
            apply_panel<CW, 1>(g, bbuf(b), b, q, lr, pk, zp, sh.bc[1], tid, kBarB, bpar);
            bar_group<CW>(kBarB);
          }
          if (which == 0) {
            // CTA 0's buffer of block b held panel b-3: wait until its storer is done with it
            if (b >= 3 && !grp_wait_cl(&ps.mb_afree[(b - 3) % kRing], ring_parity(b - 3, kRing), kBarB)) {
              ok = false;
              break;
            }
            const double *s = bbuf(b);
            const double *d = buf(b);
            const int tot = kNB * (int)g.ldab;
            for (int e = 2 * tid; e + 1 < tot; e += 2 * kCT) cl_st2(cl_map(d + e, 0), s[e], s[e + 1]);
            if ((tot & 1) && tid == 0) cl_st1(cl_map(d + tot - 1, 0), s[tot - 1]);
            __syncwarp();
            if (lane == 0) cl_arrive(&ps.mb_blk[(b - 2) % kRing], 0);  // one arrival per warp
            bar_group<CW>(kBarB);
            if (tid == 0) mbar_arrive(&ps.mb_bsent[(b - 2) % kBBufs]);  // the buffer may take block b+4
          }
        }
      }
    } else if (warp == kCW) {
      // ---------------- CTA 1, loader: blocks b >= 2 into its buffers ----------------
      for (int b = 2; b < g.npan; ++b) {
        const int e = b - 2;
        if (e >= kBBufs) {  // the buffer held block b-4, sent to CTA 0 by now
          unsigned long long *mb = &ps.mb_bsent[e % kBBufs];
          const unsigned par = ring_parity(e - kBBufs, kBBufs);
          if (!io_wait([&] { return mbar_try_wait(mb, par); }, err)) break;
        }
        double *dst = bbuf(b);
        unsigned long long *ml = &ps.mb_bload[e % kBBufs];
        if (handed_off_pair(g, b)) {
          const int *f = block_ready + b;
          if (!io_wait([&] { return ld_acquire(f) != 0; }, err)) break;
          if (g.vec && (b + 1) * kNB <= g.n) {
            if (lane == 0) bulk_prefetch_block(g, AB, dst, b, ml);  // completes the phase itself
            __syncwarp();
            continue;
          }
          if (g.vec) {
            io_prefetch_block(g, AB, dst, b);
          } else {
            load_block(g, AB, dst, b, false, lane, 32);
          }
        } else {
          load_block(g, AB, dst, b, true, lane, 32);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(ml);
      }
    }
  } else {
    // ---------------- update CTAs: panels p_first(b)..b-kHand to their blocks ----------------
    if (warp >= kCW) return;
    const int G = gridDim.x - 2, u = blockIdx.x - 2;
    int bpar = 0;
    for (int p = 0; p + kHand < g.npan; ++p) {
      const int lo = p + kHand, hi = b_last(g, p);
      const int b0 = lo + ((u - (lo - kHand)) % G + G) % G;
      if (b0 > hi) continue;
      const int *f = panel_ready + p;
      if (!compute_wait<CW, 1>([&] { return ld_acquire(f) != 0; }, err, sh)) break;
      const int c0q = p * kNB, ncq = min(kNB, g.n - c0q);
      if (tid < kNB) {
        const int k = tid;
        sh.pk[0][k] = k < ncq ? __ldcg(ipiv + c0q + k) - 1 - (c0q + k) : 0;
        sh.zp[0][k] = k < ncq ? (nz(__ldcg(AB + (long long)(c0q + k) * g.ldab + g.kv)) ? 0 : 1) : 1;
      }
      double lr[1][kNB];
#pragma unroll
      for (int k = 0; k < kNB; ++k) {
        const int t = tid - k;
        lr[0][k] = (k < ncq && t >= 1 && t <= min(g.kl, g.n - 1 - (c0q + k)))
                       ? __ldcg(AB + (long long)(c0q + k) * g.ldab + g.kv + t)
                       : 0.0;
      }
      bar_compute<CW>();
      for (int b = b0; b <= hi; b += G) {
        double *blk = blocks + (long long)(((b - kHand) / G) % kMaxActive) * bsz;
        if (p == p_first(g, b)) {
          load_block(g, AB, blk, b, true, tid, kCT);
          bar_compute<CW>();
        }
        apply_panel<CW, 1>(g, blk, b, p, lr, sh.pk[0], sh.zp[0], sh.bc[0], tid, kBarA, bpar);
        bar_compute<CW>();
        if (p == b - kHand) {
          store_block(g, AB, blk, b, tid, kCT);
          __threadfence();
          bar_compute<CW>();
          if (tid == 0) st_release(block_ready + b, 1);
        }
      }
    }
    return;
  }
  // the cluster's two CTAs leave together: no distributed-shared-memory access can
  // reach a CTA that has exited
  cluster_barrier();
}

template <int CW>
struct PairLaunch {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[2];
  // BANDLU_OK: the grid can be made resident (all clusters at once); BANDLU_NOT_BANDED:
  // it cannot (the caller takes another kernel); BANDLU_ERR_CUDA.  The occupancy answer
  // is cached per (device, grid, shared memory), so a call made during stream capture
  // after a first call outside it issues no query.
  int prepare(int grid, size_t smem, cudaStream_t s) {
    if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_gbtrf_wide_pair<CW>), 200 * 1024))
      return BANDLU_ERR_CUDA;
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(32 * (CW + 1));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeCooperative;
    at[1].val.cooperative = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return BANDLU_ERR_CUDA;
    static std::mutex mu;
    static std::map<std::tuple<int, int, size_t>, int> fits;
    const auto key = std::make_tuple(dev, grid, smem);
    {
      std::lock_guard<std::mutex> lock(mu);
      const auto it = fits.find(key);
      if (it != fits.end()) return it->second;
    }
    int clusters = 0;
    int rc = BANDLU_OK;
    if (cudaOccupancyMaxActiveClusters(&clusters, k_gbtrf_wide_pair<CW>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      rc = BANDLU_NOT_BANDED;
    } else if (clusters * 2 < grid) {
      rc = BANDLU_NOT_BANDED;
    }
    std::lock_guard<std::mutex> lock(mu);
    fits[key] = rc;
    return rc;
  }
  int launch(const Geo &g, double *AB, int *ipiv, int *d_info, int *flags, const int *d_kl, const int *d_ku) {
    cfg.attrs = at;
    cfg.numAttrs = 2;
    Geo gg = g;
    if (cudaLaunchKernelEx(&cfg, k_gbtrf_wide_pair<CW>, gg, AB, ipiv, d_info, flags, d_kl, d_ku) != cudaSuccess)
      return BANDLU_ERR_CUDA;
    return BANDLU_OK;
  }
};

template <int CW>
int launch_pair(const Geo &g, int grid, size_t smem, double *AB, int *ipiv, int *d_info, int *flags, cudaStream_t s) {
  PairLaunch<CW> pl;
  const int rc = pl.prepare(grid, smem, s);
  if (rc != BANDLU_OK) return rc;
  return pl.launch(g, AB, ipiv, d_info, flags, nullptr, nullptr);
}

template <int CW>
int pair_fits(int grid, size_t smem, cudaStream_t s) {
  PairLaunch<CW> pl;
  return pl.prepare(grid, smem, s);
}

// Shared memory of the pair kernel for band storage ldab and (largest) kl.
size_t pair_smem(long long ldab, long long kl) {
  const size_t need_a = (size_t)kPanelBufs * kNB * (size_t)ldab + (size_t)kRB * kNB * (size_t)kl;
  const size_t need_b = (size_t)kBBufs * kNB * (size_t)ldab;
  const size_t need_u = (size_t)kMaxActive * kNB * (size_t)ldab;
  return std::max(need_a, std::max(need_b, need_u)) * sizeof(double);
}

#include "gbtrf_wide_stream.cuh"

// BANDLU_WIDE_SINGLE=1 in the environment selects the single-CTA panel kernel
// for every shape (read once): the comparison the cluster pair is measured against.
bool pair_disabled() {
  static const bool off = [] {
    const char *v = std::getenv("BANDLU_WIDE_SINGLE");
    return v != nullptr && v[0] == '1';
  }();
  return off;
}

// Returns BANDLU_OK after a launch, BANDLU_NOT_BANDED when the kernel cannot be
// made resident (the caller then takes another kernel), or BANDLU_ERR_CUDA.
template <int CW, int RPT>
int launch_rpt(const Geo &g, int grid, size_t smem, double *AB, int *ipiv, int *d_info, int *flags, cudaStream_t s) {
  constexpr int kThreads = Lay<CW>::kThreads;
  if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_gbtrf_wide<CW, RPT>), 200 * 1024)) return BANDLU_ERR_CUDA;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_gbtrf_wide<CW, RPT>, kThreads, smem) != cudaSuccess)
    return BANDLU_ERR_CUDA;
  if (per_sm < 1) return BANDLU_NOT_BANDED;
  Geo gg = g;
  void *args[] = {&gg, &AB, &ipiv, &d_info, &flags};
  if (cudaLaunchCooperativeKernel((const void *)k_gbtrf_wide<CW, RPT>, dim3(grid), dim3(kThreads), args, smem, s) !=
      cudaSuccess)
    return BANDLU_ERR_CUDA;
  return BANDLU_OK;
}

}  // namespace

// Launch conditions: kv >= 2*kNB, at most 4 panel rows per compute thread (of 9 warps),
// shared memory for three blocks and two panels of multipliers, and an update
// CTA never holding more than kMaxActive blocks.  *used = false when the shape
// does not qualify (the caller then takes another kernel).
int launch_gbtrf_wide(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t s,
                      bool *used) {
  *used = false;
  const long long kv = (long long)kl + ku;
  if (n < 4 * kNB || n > INT_MAX / 2 || kl < 1 || kv < 2 * kNB || ldab > INT_MAX / kNB) return BANDLU_OK;
  // compute group: the fewest warps (2, 4 or 9) giving every panel row a thread,
  // else 9 warps with 2 or 4 rows per thread
  const int rows = kl + kNB;
  const int cw = rows <= 64 ? 2 : (rows <= 128 ? 4 : 9);
  const int rpt = (rows + 32 * cw - 1) / (32 * cw);
  if (rpt > 4) return BANDLU_OK;
  const size_t smem = ((size_t)kPanelBufs * kNB * (size_t)ldab + 2 * (size_t)kNB * kl) * sizeof(double);
  if (smem > 200 * 1024) return BANDLU_OK;
  int dev = 0, sms = 0, coop = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (!coop || sms < 2) return BANDLU_OK;
  const int G = sms - 1;
  const long long span = (kv + 3) / kNB + 1;  // blocks one panel updates, at most
  if (span > (long long)kMaxActive * G) return BANDLU_OK;
  Geo g;
  g.n = (int)n;
  g.kl = kl;
  g.ku = ku;
  g.kv = (int)kv;
  g.ldab = ldab;
  g.npan = (int)((n + kNB - 1) / kNB);
  g.vec = (reinterpret_cast<uintptr_t>(AB) & 15u) == 0;
  // scratch: error flag, spare, panel_ready[npan], block_ready[npan]
  const size_t fbytes = (size_t)(2 + 2 * (size_t)g.npan) * sizeof(int);
  int *flags = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&flags), fbytes, s) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaMemsetAsync(flags, 0, fbytes, s) != cudaSuccess) {
    cudaFreeAsync(flags, s);
    return BANDLU_ERR_CUDA;
  }
  int rc = BANDLU_NOT_BANDED;
  if (rpt == 1 && sms >= 4 && !pair_disabled()) {
    if (!chain_disabled()) {
      // the chain: CTA 0 factors, kStreamers CTAs apply the lookahead panels as they stream in
      const size_t smemc = stream_smem(ldab, cw);
      if (smemc <= 200 * 1024) {
        auto run = [&](auto &sl) {
          const int gc = sl.prepare(sms, smemc, s);
          if (gc < 0) return BANDLU_ERR_CUDA;
          if (gc == 0 || span > (long long)kMaxActive * (gc - kChainCTAs)) return BANDLU_NOT_BANDED;
          return sl.launch(g, AB, ipiv, d_info, flags, nullptr, nullptr);
        };
        if (cw == 2) {
          StreamLaunch<2> sl;
          rc = run(sl);
        } else if (cw == 4) {
          StreamLaunch<4> sl;
          rc = run(sl);
        } else {
          StreamLaunch<9> sl;
          rc = run(sl);
        }
      }
    }
    // the cluster pair: CTA 0 factors and looks ahead, CTA 1 runs the second lookahead group
    const int grid2 = sms & ~1;
    const size_t smem2 = pair_smem(ldab, kl);
    if (rc == BANDLU_NOT_BANDED && smem2 <= 200 * 1024 && span <= (long long)kMaxActive * (grid2 - 2)) {
      if (cw == 2)
        rc = launch_pair<2>(g, grid2, smem2, AB, ipiv, d_info, flags, s);
      else if (cw == 4)
        rc = launch_pair<4>(g, grid2, smem2, AB, ipiv, d_info, flags, s);
      else
        rc = launch_pair<9>(g, grid2, smem2, AB, ipiv, d_info, flags, s);
    }
  }
  if (rc != BANDLU_NOT_BANDED) {
    // launched (or failed): nothing more to do
  } else if (cw == 2)
    rc = launch_rpt<2, 1>(g, sms, smem, AB, ipiv, d_info, flags, s);
  else if (cw == 4)
    rc = launch_rpt<4, 1>(g, sms, smem, AB, ipiv, d_info, flags, s);
  else if (rpt == 1)
    rc = launch_rpt<9, 1>(g, sms, smem, AB, ipiv, d_info, flags, s);
  else if (rpt == 2)
    rc = launch_rpt<9, 2>(g, sms, smem, AB, ipiv, d_info, flags, s);
  else
    rc = launch_rpt<9, 4>(g, sms, smem, AB, ipiv, d_info, flags, s);
  if (cudaFreeAsync(flags, s) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (rc == BANDLU_NOT_BANDED) return BANDLU_OK;
  if (rc != BANDLU_OK) return rc;
  *used = true;
  return BANDLU_OK;
}

int prepare_gbtrf_wide_deferred(int64_t n, int64_t ldab, cudaStream_t s, WideDeferred *wd) {
  *wd = WideDeferred();
  if (pair_disabled() || n < 4 * kNB || n > INT_MAX / 2 || ldab > INT_MAX / kNB) return BANDLU_OK;
  // the compute group is sized for the largest kl the storage admits (up to 9 warps;
  // bands wider than the group keep the single-CTA fallback of the on-device kernel)
  const long long kl_max = (ldab - 1) / 2;
  const long long rows_max = kl_max + kNB;
  const int cw = rows_max <= 64 ? 2 : (rows_max <= 128 ? 4 : 9);
  const long long kl_cap = std::min(kl_max, (long long)32 * cw - kNB);
  int dev = 0, sms = 0, coop = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (!coop || sms < 4) return BANDLU_OK;
  const long long span_max = (ldab - 1 + 3) / kNB + 1;  // kv <= ldab - 1
  int grid = 0;
  size_t smem = 0;
  bool chain = false;
  if (!chain_disabled() && stream_smem(ldab, cw) <= 200 * 1024) {
    // the chain, as in launch_gbtrf_wide
    const size_t smemc = stream_smem(ldab, cw);
    int gc = 0;
    if (cw == 2) {
      StreamLaunch<2> sl;
      gc = sl.prepare(sms, smemc, s);
    } else if (cw == 4) {
      StreamLaunch<4> sl;
      gc = sl.prepare(sms, smemc, s);
    } else {
      StreamLaunch<9> sl;
      gc = sl.prepare(sms, smemc, s);
    }
    if (gc < 0) return BANDLU_ERR_CUDA;
    if (gc > 0 && span_max <= (long long)kMaxActive * (gc - kChainCTAs)) {
      chain = true;
      grid = gc;
      smem = smemc;
    }
  }
  if (!chain) {
    grid = sms & ~1;
    if (span_max > (long long)kMaxActive * (grid - 2)) return BANDLU_OK;
    smem = pair_smem(ldab, kl_cap);
    if (smem > 200 * 1024) return BANDLU_OK;
    const int fit =
        cw == 2 ? pair_fits<2>(grid, smem, s) : (cw == 4 ? pair_fits<4>(grid, smem, s) : pair_fits<9>(grid, smem, s));
    if (fit == BANDLU_NOT_BANDED) return BANDLU_OK;
    if (fit != BANDLU_OK) return fit;
  }
  const long long npan = (n + kNB - 1) / kNB;
  const size_t fbytes = (size_t)(2 + 2 * npan) * sizeof(int);
  int *flags = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&flags), fbytes, s) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaMemsetAsync(flags, 0, fbytes, s) != cudaSuccess) {
    cudaFreeAsync(flags, s);
    return BANDLU_ERR_CUDA;
  }
  wd->rows_cap = 32 * cw;
  wd->cw = cw;
  wd->chain = chain;
  wd->grid = grid;
  wd->smem = smem;
  wd->flags = flags;
  return BANDLU_OK;
}

int launch_gbtrf_wide_deferred(const WideDeferred &wd, int64_t n, double *AB, int64_t ldab, int *ipiv,
                               const int *d_kl, const int *d_ku, int *d_info, cudaStream_t s) {
  Geo g;
  g.n = (int)n;
  g.kl = g.ku = g.kv = 0;  // read on the device
  g.ldab = ldab;
  g.npan = (int)((n + kNB - 1) / kNB);
  g.vec = (reinterpret_cast<uintptr_t>(AB) & 15u) == 0;
  int rc = BANDLU_ERR_CUDA;
  if (wd.chain) {
    auto run = [&](auto &sl) {
      return sl.prepare(device_sms(), wd.smem, s) == wd.grid ? sl.launch(g, AB, ipiv, d_info, wd.flags, d_kl, d_ku)
                                                             : BANDLU_ERR_CUDA;
    };
    if (wd.cw == 2) {
      StreamLaunch<2> sl;
      rc = run(sl);
    } else if (wd.cw == 4) {
      StreamLaunch<4> sl;
      rc = run(sl);
    } else {
      StreamLaunch<9> sl;
      rc = run(sl);
    }
  } else if (wd.cw == 2) {
    PairLaunch<2> pl;
    if (pl.prepare(wd.grid, wd.smem, s) == BANDLU_OK) rc = pl.launch(g, AB, ipiv, d_info, wd.flags, d_kl, d_ku);
  } else if (wd.cw == 4) {
    PairLaunch<4> pl;
    if (pl.prepare(wd.grid, wd.smem, s) == BANDLU_OK) rc = pl.launch(g, AB, ipiv, d_info, wd.flags, d_kl, d_ku);
  } else {
    PairLaunch<9> pl;
    if (pl.prepare(wd.grid, wd.smem, s) == BANDLU_OK) rc = pl.launch(g, AB, ipiv, d_info, wd.flags, d_kl, d_ku);
  }
  if (cudaFreeAsync(wd.flags, s) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  return rc;
}

}  // namespace bandlu

// ---- timeline of the traced build (include/bandlu_trace.h) ----
extern "C" {

int bandlu_trace_capacity(void) {
#ifdef BANDLU_TRACE
  return bandlu::kTrPanels;
#else
  return 0;
#endif
}

int bandlu_trace_read(uint64_t *host, int64_t count) {
#ifdef BANDLU_TRACE
  if (host == nullptr) return -1;
  if (count < 0 || count > 4ll * bandlu::kTrPanels * bandlu::kTrSlots) return -2;
  if (count == 0) return BANDLU_OK;
  return cudaMemcpyFromSymbol(host, bandlu::g_chain_trace, (size_t)count * sizeof(uint64_t)) == cudaSuccess
             ? BANDLU_OK
             : BANDLU_ERR_CUDA;
#else
  (void)host;
  (void)count;
  return BANDLU_ERR_CUDA;
#endif
}

int bandlu_trace_clear(void) {
#ifdef BANDLU_TRACE
  void *p = nullptr;
  if (cudaGetSymbolAddress(&p, bandlu::g_chain_trace) != cudaSuccess) return BANDLU_ERR_CUDA;
  return cudaMemset(p, 0, sizeof(bandlu::g_chain_trace)) == cudaSuccess ? BANDLU_OK : BANDLU_ERR_CUDA;
#else
  return BANDLU_ERR_CUDA;
#endif
}

}  // extern "C"
