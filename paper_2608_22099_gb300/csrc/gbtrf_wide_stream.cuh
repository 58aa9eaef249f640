// gbtrf_wide_stream.cuh -- the wide-band factorisation (Sec. II-A step 3; f(N) ~
// O(N*P*Q), Eq. S-N-N3) with the lookahead taken off the panel CTA and streamed
// down a chain of CTAs.  Included by gbtrf_wide.cu inside its anonymous
// namespace (it uses that file's block transfers, step functions and bounded
// waits).
//
// Cluster 0 holds 1 + kStreamers CTAs:
//
//  * CTA 0 (A) only factors: block p arrives with panels 0..p-1 applied, group A
//    factors it, and after every column step each thread sends its row's
//    multiplier (thread 0 also the step's pivot offset and zero flag) into
//    streamer 1's shared memory with one 8-byte st.async, completing a
//    transaction count on streamer 1's barrier of the step.  A forwarder warp on
//    streamer r (r < kStreamers) passes each step's records on to streamer r+1
//    with one bulk copy once they have arrived: only streamer 1 is on A's path
//    (its block comes back next), the others have a panel or more in hand.  A
//    storer warp writes finished panels to AB and publishes them.
//  * In a column step only the next column's update is on the path to the
//    next pivot search; the step's update of the columns after it is issued in
//    the next step, beside its reciprocal and argmax (integer and FP32 work),
//    before anything reads those columns.
//  * Streamer 1 applies the first kNB-1 steps of panel p to block p+1; the
//    last one is applied by A as it starts panel p+1, straight from the block
//    that arrived: each thread reads the step's pivot row and row j from shared
//    memory and takes its own row's multiplier from the thread that held that
//    row in panel p (four rows lower), updates column 0 at once and the other
//    columns through the deferred update of step 0.
//  * CTA r (streamer r, 1 <= r <= kStreamers) receives every block b from CTA
//    r+1 (streamer kStreamers from its loader, which takes the block from AB once
//    an update CTA has applied panels p_first(b)..b-kHandChain), applies panel
//    b-r to it as that panel's steps arrive (the pivot row and row j broadcast
//    inside the CTA, which holds the whole block), and passes the block to CTA
//    r-1: a sender warp moves the rows the panel leaves unchanged as soon as the
//    block is in and the destination is free (bulk copies of the runs between
//    the bands), so the group goes straight to the steps, and the group sends
//    the panel's band rows from registers after the last step.  While A factors panel p, streamer
//    r applies panel p to block p+r, so each block reaches A with panels up to
//    p-1 applied, at most one step after A's last step plus one copy.
//  * The other CTAs (update CTAs) apply panels p_first(b)..b-kHandChain and hand
//    block b over (block_ready[b]).
//
// Panels are applied to a block in increasing order by whichever CTA holds it,
// with the step functions of the other kernels, so the factors are
// bit-identical to the unblocked elimination.  Rings without credits: the step
// records of panel p overwrite those of panel p-kRecDepth, which every streamer
// has read before A can hold block p (each streamer has passed block p on, after
// reading panel p-kStreamers); a block goes into a slot whose previous block
// (b-kSlots) A has already factored (panel_ready).  Every wait is bounded.
#pragma once

// Timeline of the traced build (include/bandlu_trace.h): the global timer at panel
// boundaries and waits; nothing in the production build.
constexpr int kTrPanels = 8192, kTrSlots = 16;
#ifdef BANDLU_TRACE
__device__ unsigned long long g_chain_trace[4][kTrPanels][kTrSlots];
__device__ __forceinline__ void tr_stamp(int role, int q, int slot) {
  if (q >= 0 && q < kTrPanels) {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    g_chain_trace[role][q][slot] = t;
  }
}
#define TR_STAMP(cond, role, q, slot) \
  do {                                \
    if (cond) tr_stamp(role, q, slot); \
  } while (0)
#else
#define TR_STAMP(cond, role, q, slot) \
  do {                                \
  } while (0)
#endif

constexpr int kStreamers = 4;                    // streamer CTAs after A
constexpr int kChainCTAs = kStreamers + 1;       // cluster size
constexpr int kRecDepth = kStreamers + 1;        // panels of step records per streamer
constexpr int kSlots = kStreamers + 2;           // block slots per streamer
constexpr int kHandChain = kStreamers + 1;       // update CTAs hand block b over after panel b-kHandChain

template <int CW>
struct StreamShared {
  WideShared<CW, 1> w;
  unsigned long long mb_rec[kRecDepth * kNB];  // streamer: step (q, k) arrived (1 arrival + bytes), event q / kRecDepth
  unsigned long long mb_in[kSlots];            // streamer: block b in slot (b-1) % kSlots, event (b-1) / kSlots
  unsigned long long mb_blk[kRing];            // A: block b >= 1 arrived (1 arrival + bytes), event b-1
  unsigned long long mb_afree[kRing];          // streamer 1: A's buffer of block p stored (A's storer), event p
  unsigned long long mb_pub[kRing];            // A: panel p published (publisher), event p
  unsigned long long mb_dst[kSlots];           // streamer: block b's destination free and its unchanged
                                               // rows sent (sender), event (b-1) / kSlots
  alignas(16) unsigned long long rhdr[kRecDepth * kNB][2];  // streamer: pivot offset and zero flag of (q, k)
  double lm[32 * CW];  // A: each thread's multiplier of the last step of the panel just factored
  // streamer: every thread's row of the block before a step (the step's pivot row and row j
  // are read from here), by step parity
  double rows[2][32 * CW][kNB];
  unsigned rmask[2][32 * CW];
};

__device__ __forceinline__ unsigned long long dbl_bits_w(double x) {
  return (unsigned long long)__double_as_longlong(x);
}
__device__ __forceinline__ void st_async_b64(unsigned raddr, unsigned long long v, unsigned rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b64 [%0], %1, [%2];" ::"r"(raddr), "l"(v),
               "r"(rbar)
               : "memory");
}
__device__ __forceinline__ void st_async_v2(unsigned raddr, unsigned long long a, unsigned long long b,
                                            unsigned rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.b64 [%0], {%1, %2}, [%3];" ::"r"(raddr),
               "l"(a), "l"(b), "r"(rbar)
               : "memory");
}
__device__ __forceinline__ void mbar_expect_tx_local(unsigned long long *bar, unsigned bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes) : "memory");
}

// The group's barrier, returning true iff every thread of the group passes ok.
template <int CW>
__device__ __forceinline__ bool bar_and_group(int id, bool ok) {
  unsigned r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(ok ? 1u : 0u), "r"(id), "n"(Lay<CW>::kCT)
      : "memory");
  return r != 0;
}

// I/O warp wait: every lane polls the same condition, so the warp never diverges
// around the wait; the outcome is made uniform.
template <class F>
__device__ __forceinline__ bool io_wait_all(F ready, int *err) {
  const bool ok = bounded_poll(ready, err);
  return __all_sync(FULL, ok);
}

// Where the records of panel p go on streamer 1 (cluster addresses); send: block
// p+1 exists, so streamer 1 (and its forwarder) takes panel p.
struct RecTarget {
  unsigned rec;  // multiplier slots of step 0 (step k: + k * kCT * 8)
  unsigned hdr;  // header of step 0 (step k: + k * 16)
  unsigned bar;  // barrier of step 0 (step k: + k * 8)
  bool send;
};

// factor_panel for one row per thread, streaming each step's multipliers to the streamers.
// fuse: block p holds panels 0..p-1 but for the last step of panel p-1, which is
// applied here (multipliers in lm, pivot offset and zero flag in sh.pk / sh.zp of
// panel p-1).  On return lm holds this panel's last-step multipliers.
template <int CW>
__device__ void factor_panel_stream(const Geo &g, double *blk, int p, WideShared<CW, 1> &sh, int &bpar, int &info,
                                    const RecTarget &rt, double *__restrict__ AB, int *__restrict__ ipiv,
                                    double *lm, bool fuse) {
  constexpr int kCT = Lay<CW>::kCT, kCW = CW;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c0 = p * kNB, nc = min(kNB, g.n - c0);
  const int ldab = (int)g.ldab;
  const int pp = p & 1;
  const int i = tid, row = c0 + i;
  const bool mine = i < g.kl + kNB && row < g.n;
  double *abp = AB + (long long)c0 * g.ldab;
  double v[kNB];
#pragma unroll
  for (int k = 0; k < kNB; ++k) v[k] = (mine && k < nc && i - k <= g.kl) ? blk[k * ldab + g.kv + i - k] : 0.0;
  // the previous step's multiplier, pivot row and its nonzero mask, for its deferred update
  // of the columns after the next one (pact: this row took that update)
  double pl = 0.0, pu[kNB];
  unsigned pum = 0u;
  bool pact = false;
#pragma unroll
  for (int d = 0; d < kNB; ++d) pu[d] = 0.0;
  // panel p-1's last step (row jq = c0-1, pivot row jq+pq): interchange, then the update of
  // rows jq+1..jq+kmq, i.e. threads 0..kmq-1 (held by threads 4..kmq+3 in panel p-1)
  bool wrow = false;  // row jq of this block takes the pivot row (written after step 0's barrier)
  double uq[kNB];
#pragma unroll
  for (int d = 0; d < kNB; ++d) uq[d] = 0.0;
  if (fuse && !sh.zp[(p - 1) & 1][kNB - 1]) {  // uniform
    const int pq = sh.pk[(p - 1) & 1][kNB - 1];
    const int kmq = min(g.kl, g.n - c0);
    double r0[kNB];
#pragma unroll
    for (int d = 0; d < kNB; ++d) {
      uq[d] = d < nc ? blk[d * ldab + g.kv + pq - 1 - d] : 0.0;
      r0[d] = d < nc ? blk[d * ldab + g.kv - 1 - d] : 0.0;
    }
    if (pq != 0 && i == pq - 1) {
#pragma unroll
      for (int d = 0; d < kNB; ++d) v[d] = r0[d];
    }
    wrow = pq != 0;
    if (i < kmq) {
      const double l = lm[i + kNB];
      const unsigned um = nz_mask(uq);
      v[0] = upd(l, uq[0], v[0], um & 1u);
      pl = l;
      pact = true;
#pragma unroll
      for (int d = 0; d < kNB; ++d) pu[d] = uq[d];
      pum = um;
    }
  }
  double lastl = 0.0;
#pragma unroll
  for (int k = 0; k < kNB; ++k) {
    if (k >= nc) break;
    const int j = c0 + k, km = min(g.kl, g.n - 1 - j);
    const int s = bpar;
    bpar ^= 1;
    TR_STAMP(tid == 0, 0, p, 4 + 3 * k);
    const int t = i - k;
    bool myspec;
    const double myr = rcp_rn_fast(v[k], &myspec);
    const unsigned long long key = (t >= 0 && t <= km) ? pivot_key(v[k], t == 0) : 0ull;
    // step k-1's update of columns k+1.. (its update of column k is done): before this
    // step publishes or interchanges anything, so every element still receives the
    // steps in order
    if (pact) {
#pragma unroll
      for (int d = 0; d < kNB; ++d)
        if (d > k) v[d] = upd(pl, pu[d], v[d], (pum >> d) & 1u);
    }
    unsigned long long kmax;
    const int wl = warp_first_max(key, &kmax);
    if (lane == wl) {
      sh.key[s][warp] = kmax;
      sh.idx[s][warp] = i;
#pragma unroll
      for (int d = 0; d < kNB; ++d) sh.piv[s][warp][d] = v[d];
      sh.pivm[s][warp] = nz_mask(v);
      sh.prc[s][warp] = myr;
      sh.pspec[s][warp] = myspec ? 1 : 0;
    }
    if (i == k) {
#pragma unroll
      for (int d = 0; d < kNB; ++d) sh.row0[s][d] = v[d];
    }
    bar_compute<CW>();
    TR_STAMP(tid == 0, 0, p, 5 + 3 * k);
    if (k == 0 && wrow && tid == 0) {  // every thread has read row jq above
#pragma unroll
      for (int d = 0; d < kNB; ++d)
        if (d < nc) blk[d * ldab + g.kv - 1 - d] = uq[d];
    }
    int wb = 0;
    if constexpr (kCW <= 32) {
      const unsigned long long kx = lane < kCW ? sh.key[s][lane] : 0ull;
      unsigned long long kbest;
      wb = warp_first_max(kx, &kbest);
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
    double lsend = 0.0;
    lastl = 0.0;
    pact = false;
    if (!zero) {
      double rc = sh.prc[s][wb];
      if (sh.pspec[s][wb]) rc = rcp_division(u[k]);  // uniform
      if (i == k) {
#pragma unroll
        for (int d = 0; d < kNB; ++d)
          if (d >= k) v[d] = u[d];
      } else if (p_off != 0 && i == k + p_off) {
#pragma unroll
        for (int d = 0; d < kNB; ++d)
          if (d >= k) v[d] = sh.row0[s][d];
      }
      if (i > k && i <= k + km) {
        const double l = v[k] * rc;
        v[k] = l;
        lsend = l;
        lastl = l;
        if (k + 1 < kNB) v[k + 1] = upd(l, u[k + 1], v[k + 1], (um >> (k + 1)) & 1u);
        pl = l;
        pact = true;
#pragma unroll
        for (int d = 0; d < kNB; ++d) pu[d] = u[d];
        pum = um;
      }
    }
    if (rt.send) {  // uniform; streamer 1 passes every step on, and applies all but the last
      st_async_b64(rt.rec + (unsigned)(k * kCT + tid) * 8u, dbl_bits_w(lsend), rt.bar + (unsigned)k * 8u);
      if (tid == 0)
        st_async_v2(rt.hdr + (unsigned)k * 16u, (unsigned long long)(unsigned)p_off, zero ? 1ull : 0ull,
                    rt.bar + (unsigned)k * 8u);
    }
    TR_STAMP(k == 2 && tid == 0, 0, p, 1);
    TR_STAMP(tid == 0, 0, p, 6 + 3 * k);
  }
  // every column is final now (an interchange touches the columns from its own on): what the
  // update CTAs read, the diagonals and the multipliers (band rows kv..kv+kl), goes straight
  // into AB, so the publisher only has to release it once every warp has arrived
  if (mine) {
#pragma unroll
    for (int k = 0; k < kNB; ++k) {
      if (k < nc && i - k <= g.kl) {
        blk[k * ldab + g.kv + i - k] = v[k];
        if (i >= k) abp[k * ldab + g.kv + i - k] = v[k];
      }
    }
  }
  lm[tid] = lastl;  // read by panel p+1 after the group's next barrier
  if (tid == 0) {
#pragma unroll
    for (int k = 0; k < kNB; ++k)
      if (k < nc) ipiv[c0 + k] = c0 + k + sh.pk[pp][k] + 1;
  }
}

// One step k of panel q applied to the thread's row of a block (registers w),
// the pivot row and row j broadcast through bc (the step functions' order).
template <int CW>
__device__ __forceinline__ void apply_step_regs(const Geo &g, double (&w)[kNB], int i, int k, int km, int p, double l,
                                                Bcast &bc, int bar, int &bpar) {
  const int s = bpar;
  bpar ^= 1;
  if (i == k + p) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) bc.bu[s][d] = w[d];
    bc.bum[s] = nz_mask(w);
  }
  if (i == k) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) bc.br0[s][d] = w[d];
  }
  bar_group<CW>(bar);
  double u[kNB];
#pragma unroll
  for (int d = 0; d < kNB; ++d) u[d] = bc.bu[s][d];
  const unsigned um = bc.bum[s];
  if (i == k) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = u[d];
  } else if (p != 0 && i == k + p) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = bc.br0[s][d];
  }
  if (i > k && i <= k + km) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = upd(l, u[d], w[d], (um >> d) & 1u);
  }
}

// One step k of panel q on a streamer's rows (registers w), after the step's barrier:
// the pivot row and row j come from the rows every thread published before it.
template <int CW>
__device__ __forceinline__ void apply_step_published(double (&w)[kNB], int i, int k, int km, int p, double l,
                                                     const double (*rows)[kNB], const unsigned *rmask) {
  double u[kNB];
#pragma unroll
  for (int d = 0; d < kNB; ++d) u[d] = rows[k + p][d];
  const unsigned um = rmask[k + p];
  if (i == k) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = u[d];
  } else if (p != 0 && i == k + p) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = rows[k][d];
  }
  if (i > k && i <= k + km) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = upd(l, u[d], w[d], (um >> d) & 1u);
  }
}

// The same for a block's last step, handing each column's final value to send(d, x) as soon
// as it is formed, so the sends overlap the updates of the columns after it.
template <int CW, class Send>
__device__ __forceinline__ void apply_step_published_send(double (&w)[kNB], int i, int k, int km, int p, double l,
                                                          const double (*rows)[kNB], const unsigned *rmask,
                                                          Send send) {
  double u[kNB];
#pragma unroll
  for (int d = 0; d < kNB; ++d) u[d] = rows[k + p][d];
  const unsigned um = rmask[k + p];
  if (i == k) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = u[d];
  } else if (p != 0 && i == k + p) {
#pragma unroll
    for (int d = 0; d < kNB; ++d) w[d] = rows[k][d];
  }
  const bool act = i > k && i <= k + km;
#pragma unroll
  for (int d = 0; d < kNB; ++d) {
    if (act) w[d] = upd(l, u[d], w[d], (um >> d) & 1u);
    send(d, w[d]);
  }
}

// Blocks b >= kHandChain pass through an update CTA, which applies panels
// p_first(b)..b-kHandChain.
__device__ __forceinline__ bool handed_off_chain(const Geo &g, int b) {
  return b >= kHandChain && p_first(g, b) <= b - kHandChain;
}

template <int CW>
__global__ void __launch_bounds__(32 * (CW + 2), 1)
    k_gbtrf_wide_chain(Geo g0, double *__restrict__ AB, int *__restrict__ ipiv, int *__restrict__ d_info,
                       int *__restrict__ flags, const int *__restrict__ d_kl, const int *__restrict__ d_ku) {
  constexpr int kCT = Lay<CW>::kCT, kCW = CW;
  Geo g = g0;
  if (d_kl != nullptr) {
    // enqueued by the device-side dispatch: every CTA reads the decision and (kl, ku) alike
    if (*(volatile const int *)(flags + 1) == 0) return;
    g.kl = *d_kl;
    g.ku = *d_ku;
    g.kv = g.kl + g.ku;
  }
  extern __shared__ __align__(16) double smem[];
  __shared__ StreamShared<CW> ss;
  WideShared<CW, 1> &sh = ss.w;
  int *err = flags;
  int *panel_ready = flags + 2;
  int *block_ready = flags + 2 + g.npan;
  const long long bsz = (long long)kNB * g.ldab;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // A: kPanelBufs block buffers; a streamer: kSlots block slots and its step records;
  // update CTAs: kMaxActive block buffers
  double *blocks = smem;
  double *recs = smem + (size_t)kSlots * bsz;  // kRecDepth * kNB slots of kCT multipliers
  auto buf = [&](int b) { return blocks + (long long)(b % kPanelBufs) * bsz; };
  auto sbuf = [&](int b) { return blocks + (long long)((b - 1) % kSlots) * bsz; };
  auto rslot = [](int q, int k) { return (q % kRecDepth) * kNB + k; };

  if (tid == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&sh.mb_done[i], kCW);  // one arrival per warp of group A
      mbar_init(&ss.mb_blk[i], 1);
      mbar_init(&ss.mb_afree[i], 1);
      mbar_init(&ss.mb_pub[i], 1);
    }
    for (int i = 0; i < kRecDepth * kNB; ++i) mbar_init(&ss.mb_rec[i], 1);
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(&ss.mb_in[i], 1);
      mbar_init(&ss.mb_dst[i], 1);
    }
    sh.info = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  cluster_barrier();  // every CTA's barriers initialised before any remote operation

  // a group's wait: every thread polls (a lone polling thread in an otherwise parked warp
  // is slow to see the event), one barrier makes the outcome uniform
  auto grp_wait = [&](auto ready, int bar_id) -> bool { return bar_and_group<CW>(bar_id, bounded_poll(ready, err)); };

  if (blockIdx.x == 0) {
    if (warp < kCW) {
      // ---------------- A, group: panel p factored, its steps streamed to the streamers ----------------
      int info = 0, bpar = 0;
      load_block(g, AB, buf(0), 0, true, tid, kCT);
      bar_compute<CW>();
      for (int p = 0; p < g.npan; ++p) {
        // block p+1 arrives from streamer 1 once panel p is applied to it
        if (tid == 0 && p + 1 < g.npan)
          mbar_expect_tx_local(&ss.mb_blk[p % kRing],
                               (unsigned)(min(kNB, g.n - (p + 1) * kNB) * g.ldab * (long long)sizeof(double)));
        RecTarget rt;
        rt.rec = cl_map(recs + (size_t)rslot(p, 0) * kCT, 1);
        rt.hdr = cl_map(&ss.rhdr[rslot(p, 0)][0], 1);
        rt.bar = cl_map(&ss.mb_rec[rslot(p, 0)], 1);
        rt.send = p + 1 < g.npan;  // streamer 1 applies panel p to block p+1
        TR_STAMP(tid == 0, 0, p, 0);
        factor_panel_stream<CW>(g, buf(p), p, sh, bpar, info, rt, AB, ipiv, ss.lm, p > 0);
        if (tid == 0) {
          sh.info = info;
#pragma unroll
          for (int k = 0; k < kNB; ++k) sh.pvr[p % kRing][k] = sh.pk[p & 1][k];
        }
        // the publisher and the storer: each warp arrives once its stores are issued (the
        // arrival releases them); the next panel's reads of lm and sh.pk are ordered by the
        // barrier of the wait for block p+1
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.mb_done[p % kRing]);
        TR_STAMP(tid == 0, 0, p, 2);
        if (p + 1 < g.npan) {
          unsigned long long *mb = &ss.mb_blk[p % kRing];
          const unsigned par = ring_parity(p, kRing);
          if (!grp_wait([&] { return cl_try_wait(mb, par); }, kBarA)) break;
          TR_STAMP(tid == 0, 0, p, 3);
          // block p+1 holds panel p's steps but the last, which the next factor_panel_stream applies
        }
      }
    } else if (warp == kCW) {
      // ---------------- A, publisher: panel p's diagonal, multipliers and pivots released ----------------
      // group A stored them to AB before its arrival on mb_done; that arrival (release), this
      // warp's acquire and the release below carry them to every CTA that acquires panel_ready
      for (int p = 0; p < g.npan; ++p) {
        unsigned long long *mb = &sh.mb_done[p % kRing];
        if (!io_wait_all([&] { return mbar_try_wait(mb, ring_parity(p, kRing)); }, err)) break;
        if (lane == 0) {
          st_release(panel_ready + p, 1);
          mbar_arrive(&ss.mb_pub[p % kRing]);
        }
        __syncwarp();
      }
    } else if (warp == kCW + 1) {
      // ---------------- A, storer: the whole finished block, then its buffer is free ----------------
      for (int p = 0; p < g.npan; ++p) {
        unsigned long long *mb = &ss.mb_pub[p % kRing];
        if (!io_wait_all([&] { return mbar_try_wait(mb, ring_parity(p, kRing)); }, err)) break;
        store_block(g, AB, buf(p), p, lane, 32);
        __syncwarp();
        // this buffer takes block p+3 next, which streamer 1 sends
        if (p + 3 < g.npan && lane == 0) cl_arrive(&ss.mb_afree[p % kRing], 1);
      }
      // info is final once the last panel is done; the status reflects every CTA's waits
      if (lane == 0) *d_info = ld_acquire(err) ? -BANDLU_ERR_TIMEOUT : sh.info;
    }
  } else if (blockIdx.x < kChainCTAs) {
    const int r = blockIdx.x;  // streamer r: panel b-r to block b, then block b to CTA r-1
    const int ld = (int)g.ldab;
    const int boff = g.kv - kNB * r;  // band position of row 4(b-r), column 0
    // where block b goes: A's buffer (which held block b-3: its storer must be done), or
    // streamer r-1's slot (which held block b-kSlots: A must have factored it)
    auto dest = [&](int b, unsigned &dst, unsigned &dbar) {
      if (r == 1) {
        dst = cl_map(buf(b), 0);
        dbar = cl_map(&ss.mb_blk[(b - 1) % kRing], 0);
      } else {
        dst = cl_map(sbuf(b), r - 1);
        dbar = cl_map(&ss.mb_in[(b - 1) % kSlots], r - 1);
      }
    };
    auto applies = [&](int b) { return b - r >= 0 && b - r >= p_first(g, b); };
    const int sender = r < kStreamers ? kCW : kCW + 1;
    if (warp < kCW) {
      int bpar = 0;
      const int i = tid;
      for (int b = 1; b < g.npan; ++b) {
        const int slot = (b - 1) % kSlots;
        const int c0b = b * kNB, ncb = min(kNB, g.n - c0b);
        const unsigned bytes = (unsigned)(ncb * ld * 8);  // what a block's move carries
        if (r < kStreamers && tid == 0) mbar_expect_tx_local(&ss.mb_in[slot], bytes);
        {
          unsigned long long *mb = &ss.mb_in[slot];
          const unsigned par = ring_parity(b - 1, kSlots);
          if (!grp_wait([&] { return cl_try_wait(mb, par); }, kBarB)) break;
        }
        TR_STAMP(r <= 2 && tid == 0, r, b - r, 0);
        const int q = b - r;
        const bool apply = applies(b);  // uniform
        double *bx = sbuf(b);
        unsigned dst, dbar;
        dest(b, dst, dbar);
        bool sent = false;  // the band went out within the last step
        double w[kNB];  // this thread's row of panel q's band in the block
        if (q >= 0) {
          // panel q as its steps stream from A (streamer 1 leaves the last one to A); the
          // records are taken whether or not the panel reaches this block
          const int c0q = q * kNB, ncq = min(kNB, g.n - c0q);
          const int nsteps = r == 1 ? ncq - 1 : ncq;
          const int row = c0q + i;
          const bool mine = i < g.kl + kNB && row < g.n;
#pragma unroll
          for (int d = 0; d < kNB; ++d) {
            const int pos = boff + i - d;
            w[d] = (apply && i < g.kl + kNB && d < ncb && pos >= 0 && pos < ld) ? bx[d * ld + pos] : 0.0;
          }
          bool ok = true;
#pragma unroll
          for (int k = 0; k < kNB; ++k) {
            if (k >= nsteps) break;  // uniform
            const int sl = rslot(q, k);
            // this thread's row as it stands, for the step's pivot row and row j; the wait's
            // barrier below makes every row visible (slot bpar was last read two steps ago)
            const int sb = bpar;
            bpar ^= 1;
#pragma unroll
            for (int d = 0; d < kNB; ++d) ss.rows[sb][i][d] = w[d];
            ss.rmask[sb][i] = nz_mask(w);
            // the last streamer opens its own phases; the others' forwarder has opened them
            if (r == kStreamers && tid == 0) mbar_expect_tx_local(&ss.mb_rec[sl], (unsigned)(kCT * 8 + 16));
            unsigned long long *mb = &ss.mb_rec[sl];
            const unsigned par = ring_parity(q, kRecDepth);
            TR_STAMP(r <= 2 && tid == 0 && k == nsteps - 1, r, q, 2);
            // the block's last step also takes the sender's arrival (destination free), made
            // long before, in the same wait
            unsigned long long *md = &ss.mb_dst[slot];
            const unsigned pard = ring_parity(b - 1, kSlots);
            const bool lastk = k == nsteps - 1;
            if (!grp_wait([&] { return cl_try_wait(mb, par) && (!lastk || mbar_try_wait(md, pard)); }, kBarB)) {
              ok = false;
              break;
            }
            TR_STAMP(r <= 2 && tid == 0 && k == 0, r, q, 1);
            TR_STAMP(r <= 2 && tid == 0 && k == nsteps - 1, r, q, 3);
            if (apply && !ss.rhdr[sl][1]) {  // uniform
              const double l = recs[(size_t)sl * kCT + i];
              const int pk = (int)ss.rhdr[sl][0];
              const int km = min(g.kl, g.n - 1 - (c0q + k));
              double wm[kNB];
#pragma unroll
              for (int d = 0; d < kNB; ++d) wm[d] = w[d];
              if (lastk) {
                // the block's last step here (the destination is free: taken in the wait above)
                apply_step_published_send<CW>(wm, i, k, km, pk, l, ss.rows[sb], ss.rmask[sb], [&](int d, double x) {
                  const int pos = boff + i - d;
                  if (i < g.kl + kNB && d < ncb && pos >= 0 && pos < ld)
                    st_async_b64(dst + (unsigned)(d * ld + pos) * 8u, dbl_bits_w(x), dbar);
                });
                sent = true;
                TR_STAMP(r <= 2 && tid == 0, r, q, 4);
              } else {
                apply_step_published<CW>(wm, i, k, km, pk, l, ss.rows[sb], ss.rmask[sb]);
              }
              if (mine) {
#pragma unroll
                for (int d = 0; d < kNB; ++d) w[d] = wm[d];
              }
            }
          }
          if (!ok) break;
        }
        if (!sent) {
          // the destination is free (the sender has seen it) and the unchanged rows are on their way
          unsigned long long *mb = &ss.mb_dst[slot];
          const unsigned par = ring_parity(b - 1, kSlots);
          if (!grp_wait([&] { return mbar_try_wait(mb, par); }, kBarB)) break;
        }
        if (q >= 0 && !sent) {
          // the band: one value per (row, column), from the row's thread
          if (apply && i < g.kl + kNB) {
#pragma unroll
            for (int d = 0; d < kNB; ++d) {
              const int pos = boff + i - d;
              if (d < ncb && pos >= 0 && pos < ld) st_async_b64(dst + (unsigned)(d * ld + pos) * 8u, dbl_bits_w(w[d]), dbar);
            }
          }
          TR_STAMP(r <= 2 && tid == 0, r, q, 4);
        }
      }
    } else if (warp == sender) {
      // ---------------- sender: the rows panel b-r leaves unchanged, as soon as they can go ----------------
      // Panel b-r's rows of block b (band positions boff-d .. boff+kl+3-d of column d) change in
      // the group; every other value is final and goes now.  Between the bands the block is
      // ncb+1 runs (a column's tail and the next column's head are contiguous): each a bulk copy
      // between 16-byte boundaries (lane 0), the at most one value cut off at each end as an
      // 8-byte st.async (lanes 1 and 2).  Then one arrival tells the group it may send the band.
      for (int b = 1; b < g.npan; ++b) {
        const int slot = (b - 1) % kSlots;
        const int ncb = min(kNB, g.n - b * kNB);
        {
          unsigned long long *mb = &ss.mb_in[slot];
          const unsigned par = ring_parity(b - 1, kSlots);
          if (!io_wait_all([&] { return cl_try_wait(mb, par); }, err)) break;
        }
        if (r == 1) {
          if (b >= 3) {
            unsigned long long *mb = &ss.mb_afree[(b - 3) % kRing];
            const unsigned par = ring_parity(b - 3, kRing);
            if (!io_wait_all([&] { return cl_try_wait(mb, par); }, err)) break;
          }
        } else if (b - kSlots >= 1) {
          const int *f = panel_ready + (b - kSlots);
          if (!io_wait_all([&] { return ld_acquire(f) != 0; }, err)) break;
        }
        const bool apply = applies(b);
        const double *bx = sbuf(b);
        unsigned dst, dbar;
        dest(b, dst, dbar);
        auto band = [&](int d, int &lo, int &hi) {  // band of column d, [lo, hi]; lo > hi: none
          lo = ld;
          hi = ld - 1;
          if (apply) {
            const int l0 = max(0, boff - d), h0 = min(ld - 1, boff + g.kl + kNB - 1 - d);
            if (h0 >= l0) {
              lo = l0;
              hi = h0;
            }
          }
        };
        if (lane == 0) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        for (int j = 0; j <= ncb; ++j) {
          int e0, e1;  // element range of run j
          if (j == 0) {
            int lo, hi;
            band(0, lo, hi);
            e0 = 0;
            e1 = lo;
          } else {
            int lo, hi;
            band(j - 1, lo, hi);
            e0 = (j - 1) * ld + hi + 1;
            if (j < ncb) {
              int lo2, hi2;
              band(j, lo2, hi2);
              e1 = j * ld + lo2;
            } else {
              e1 = ncb * ld;
            }
          }
          if (e1 > e0) {
            const int a0 = (e0 + 1) & ~1, a1 = e1 & ~1;  // 16-byte aligned element range
            if (a1 > a0) {
              if (lane == 0)
                asm volatile(
                    "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                        dst + (unsigned)a0 * 8u),
                    "r"(smem_addr(bx + a0)), "r"((unsigned)(a1 - a0) * 8u), "r"(dbar)
                    : "memory");
              if (lane == 1 && e0 < a0) st_async_b64(dst + (unsigned)e0 * 8u, dbl_bits_w(bx[e0]), dbar);
              if (lane == 2 && a1 < e1) st_async_b64(dst + (unsigned)a1 * 8u, dbl_bits_w(bx[a1]), dbar);
            } else {
              if (lane == 1) st_async_b64(dst + (unsigned)e0 * 8u, dbl_bits_w(bx[e0]), dbar);
              if (lane == 2 && e0 + 1 < e1) st_async_b64(dst + (unsigned)(e0 + 1) * 8u, dbl_bits_w(bx[e0 + 1]), dbar);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&ss.mb_dst[slot]);
      }
    } else if (warp == kCW + 1 && r < kStreamers) {
      // ---------------- forwarder: panel q's step records on to streamer r+1 ----------------
      // This streamer takes panel q iff block q+r exists, streamer r+1 iff block q+r+1 does.
      // This warp opens every step's phase (expect_tx) itself, so a phase completes as soon as
      // its records land, however far behind the group is, and the records move on at once.
      // Slot (q, k) held (q-5, k), whose phase this warp has seen complete; this streamer's
      // group and streamer r+1 have read (q-5, k) before A can send (q, k) (block q+5 has
      // passed through both), so both slots are free and the group's wait on (q-5, k)'s
      // parity cannot be confused with (q, k)'s.
      const unsigned rbytes = (unsigned)(kCT * 8);
      bool ok = true;
      for (int q = 0; ok && q + r < g.npan; ++q) {
        const int ncq = min(kNB, g.n - q * kNB);
        const bool fwd = q + r + 1 < g.npan;
        for (int k = 0; k < ncq; ++k) {
          const int sl = rslot(q, k);
          unsigned long long *mb = &ss.mb_rec[sl];
          if (lane == 0) mbar_expect_tx_local(mb, rbytes + 16u);
          const unsigned par = ring_parity(q, kRecDepth);
          if (!io_wait_all([&] { return cl_try_wait(mb, par); }, err)) {
            ok = false;
            break;
          }
          if (fwd && lane == 0) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            const unsigned rb = cl_map(mb, r + 1);
            asm volatile(
                "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    cl_map(recs + (size_t)sl * kCT, r + 1)),
                "r"(smem_addr(recs + (size_t)sl * kCT)), "r"(rbytes), "r"(rb)
                : "memory");
            asm volatile(
                "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    cl_map(&ss.rhdr[sl][0], r + 1)),
                "r"(smem_addr(&ss.rhdr[sl][0])), "r"(16u), "r"(rb)
                : "memory");
          }
          __syncwarp();
        }
      }
    } else if (warp == kCW && r == kStreamers) {
      // ---------------- last streamer, loader: blocks b >= 1 into its slots ----------------
      for (int b = 1; b < g.npan; ++b) {
        // the slot held block b-kSlots, passed on by now: A has factored it
        if (b - kSlots >= 1) {
          const int *f = panel_ready + (b - kSlots);
          if (!io_wait_all([&] { return ld_acquire(f) != 0; }, err)) break;
        }
        double *dst = sbuf(b);
        unsigned long long *ml = &ss.mb_in[(b - 1) % kSlots];
        if (handed_off_chain(g, b)) {
          const int *f = block_ready + b;
          TR_STAMP(lane == 0, 3, b, 0);
          if (!io_wait_all([&] { return ld_acquire(f) != 0; }, err)) break;
          TR_STAMP(lane == 0, 3, b, 1);
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
    // ---------------- update CTAs: panels p_first(b)..b-kHandChain to their blocks ----------------
    if (warp >= kCW) return;
    const int G = gridDim.x - kChainCTAs, u = blockIdx.x - kChainCTAs;
    int bpar = 0;
    for (int p = 0; p + kHandChain < g.npan; ++p) {
      const int lo = p + kHandChain, hi = b_last(g, p);
      const int b0 = lo + ((u - (lo - kHandChain)) % G + G) % G;
      if (b0 > hi) continue;
      const int *f = panel_ready + p;
      if (!bar_and_group<CW>(kBarA, bounded_poll([&] { return ld_acquire(f) != 0; }, err))) break;
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
        double *blk = blocks + (long long)(((b - kHandChain) / G) % kMaxActive) * bsz;
        if (p == p_first(g, b)) {
          load_block(g, AB, blk, b, true, tid, kCT);
          bar_compute<CW>();
        }
        apply_panel<CW, 1>(g, blk, b, p, lr, sh.pk[0], sh.zp[0], sh.bc[0], tid, kBarA, bpar);
        bar_compute<CW>();
        if (p == b - kHandChain) {
          // the block to AB, then the hand-over: the barrier orders every thread's stores before
          // thread 0's release, which (being cumulative) makes them visible with the flag
          store_block(g, AB, blk, b, tid, kCT);
          bar_compute<CW>();
          if (tid == 0) st_release(block_ready + b, 1);
        }
      }
    }
    return;
  }
  // after a wait gave up, let a bulk copy or st.async still in flight land
  if (ld_relaxed(err) != 0) {
    const long long t0 = clock64();
    while (clock64() - t0 < 4000000) {
    }
  }
  // the cluster's CTAs leave together: no distributed-shared-memory access or bulk copy
  // can reach a CTA that has exited
  cluster_barrier();
}
// Shared memory of the chain kernel: A three blocks, a streamer kSlots blocks and its
// step records, update CTAs two blocks.
size_t stream_smem(long long ldab, int cw) {
  const size_t bs = (size_t)kNB * (size_t)ldab;
  const size_t need_a = (size_t)kPanelBufs * bs;
  const size_t need_b = (size_t)kSlots * bs + (size_t)kRecDepth * kNB * 32 * (size_t)cw;
  const size_t need_u = (size_t)kMaxActive * bs;
  return std::max(need_a, std::max(need_b, need_u)) * sizeof(double);
}

// Cooperative launch with clusters of kChainCTAs.  prepare() answers with the grid: as
// many whole clusters as can be resident at once (up to sms / kChainCTAs), 0 when fewer
// than two fit, -1 on a CUDA error.  The answer is cached per (device, sms, shared
// memory), so a call made during stream capture after a first call outside it issues no
// query.
template <int CW>
struct StreamLaunch {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[2];
  int prepare(int sms, size_t smem, cudaStream_t s) {
    if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_gbtrf_wide_chain<CW>), 200 * 1024)) return -1;
    const int want = (sms / kChainCTAs) * kChainCTAs;
    if (want < 2 * kChainCTAs) return 0;
    cfg.gridDim = dim3((unsigned)want);
    cfg.blockDim = dim3(32 * (CW + 2));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = kChainCTAs;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeCooperative;
    at[1].val.cooperative = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -1;
    static std::mutex mu;
    static std::map<std::tuple<int, int, size_t>, int> grids;
    const auto key = std::make_tuple(dev, want, smem);
    int grid = 0;
    {
      std::lock_guard<std::mutex> lock(mu);
      const auto it = grids.find(key);
      if (it != grids.end()) grid = it->second;
    }
    if (grid == 0) {
      int clusters = 0;
      if (cudaOccupancyMaxActiveClusters(&clusters, k_gbtrf_wide_chain<CW>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        clusters = 0;
      }
      grid = std::min(clusters, want / kChainCTAs) * kChainCTAs;
      if (grid < 2 * kChainCTAs) grid = -2;  // cached "does not fit"
      std::lock_guard<std::mutex> lock(mu);
      grids[key] = grid;
    }
    if (grid < 0) return 0;
    cfg.gridDim = dim3((unsigned)grid);
    return grid;
  }
  int launch(const Geo &g, double *AB, int *ipiv, int *d_info, int *flags, const int *d_kl, const int *d_ku) {
    cfg.attrs = at;
    cfg.numAttrs = 2;
    Geo gg = g;
    if (cudaLaunchKernelEx(&cfg, k_gbtrf_wide_chain<CW>, gg, AB, ipiv, d_info, flags, d_kl, d_ku) != cudaSuccess)
      return BANDLU_ERR_CUDA;
    return BANDLU_OK;
  }
};

// BANDLU_WIDE_PAIR=1 in the environment selects the cluster pair where the chain would
// run (read once): the comparison the chain is measured against.
bool chain_disabled() {
  static const bool off = [] {
    const char *v = std::getenv("BANDLU_WIDE_PAIR");
    return v != nullptr && v[0] == '1';
  }();
  return off;
}
