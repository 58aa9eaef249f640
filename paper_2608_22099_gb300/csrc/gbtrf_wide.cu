// gbtrf_wide.cu -- banded LU for wide bands (kl beyond the windowed kernel):
// a persistent, cooperatively launched kernel, one CTA per SM (Sec. II-A step 3;
// f(N) ~ O(N*P*Q), Eq. S-N-N3).
//
// The columns are cut into blocks of kNB.  Block p is panel p.
//  * CTA 0 (panel CTA) factors panel p in shared memory (unblocked, the xGBTRF
//    order of operations), writes it to AB and publishes it (panel_ready[p]);
//    then it applies panel p to block p+1 (one-panel lookahead), which thereby
//    becomes panel p+1, fully updated.
//  * CTAs 1..G-1 (update CTAs) own the blocks b >= 2, block b on CTA
//    1 + (b-2) mod (G-1).  A block is read into shared memory when the first
//    panel reaching it is published, receives panels p_first(b)..b-2 in order,
//    and is handed to the panel CTA (written to AB, block_ready[b]) one panel
//    before the panel CTA needs it.
// Every entry receives exactly the fma sequence of the unblocked elimination,
// in the same order (the interchanges are the same permutations applied to
// the same values), so the factors are bit-identical to it.
//
// Hand-offs are acquire/release flags in global memory with bounded waits: a
// wait that gives up raises an error flag that every CTA checks, the kernel
// ends, and *d_info becomes -BANDLU_ERR_TIMEOUT.
#include <climits>

#include "common.cuh"
#include "rcp.cuh"

namespace bandlu {
namespace {

constexpr int kNB = 4;          // panel width = column block width
constexpr int kThreads = 256;
constexpr int kMaxActive = 2;   // blocks an update CTA holds at once
constexpr long long kSpinLimitCycles = 2000000000ll;

__device__ __forceinline__ int ld_acquire(const int *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int *p, int v) {
  asm volatile("st.release.gpu.global.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Whole CTA: thread 0 waits for *flag != 0 (bounded), the result is shared.
__device__ bool cta_wait(const int *flag, int *err, int *s_ok) {
  if (threadIdx.x == 0) {
    int ok = 1;
    const long long t0 = clock64();
    for (unsigned it = 0;; ++it) {
      if (ld_acquire(flag) != 0) break;
      if (ld_acquire(err) != 0) {
        ok = 0;
        break;
      }
      if ((it & 63u) == 63u && clock64() - t0 > kSpinLimitCycles) {
        atomicExch(err, 1);
        ok = 0;
        break;
      }
      __nanosleep(64);
    }
    *s_ok = ok;
  }
  __syncthreads();
  const bool ok = *s_ok != 0;
  __syncthreads();
  return ok;
}

// Whole CTA: make this CTA's global writes visible, then set *flag.
__device__ void cta_signal(int *flag) {
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) st_release(flag, 1);
}

struct Geo {
  int n, kl, ku, kv;
  long long ldab;
  int npan;
};

// First panel whose U rows reach block b: panel p reaches column (p+1)*kNB - 1 + kv.
__device__ __forceinline__ int p_first(const Geo &g, int b) {
  const int x = b * kNB - g.kv + 1;
  return x <= 0 ? 0 : (x + kNB - 1) / kNB - 1;
}
// Last block reached by panel p.
__device__ __forceinline__ int b_last(const Geo &g, int p) {
  return min(g.npan - 1, ((p + 1) * kNB - 1 + g.kv) / kNB);
}
__device__ __forceinline__ bool handed_off(const Geo &g, int b) { return b >= 2 && p_first(g, b) <= b - 2; }

// Block b (columns b*kNB ..) from AB into shared memory (kNB x ldab, AB layout).
// first: the block's first read, so its fill rows 0..kl-1 are cleared (the
// elimination clears every fill row before it starts).
__device__ void load_block(const Geo &g, const double *AB, double *blk, int b, bool first) {
  const int c0 = b * kNB, nc = min(kNB, g.n - c0);
  const long long tot = (long long)nc * g.ldab;
  const double *src = AB + (long long)c0 * g.ldab;
  for (long long e = threadIdx.x; e < tot; e += kThreads) {
    const long long r = e % g.ldab;
    blk[e] = (first && r < g.kl) ? 0.0 : __ldcg(src + e);
  }
  __syncthreads();
}

__device__ void store_block(const Geo &g, double *AB, const double *blk, int b) {
  const int c0 = b * kNB, nc = min(kNB, g.n - c0);
  const long long tot = (long long)nc * g.ldab;
  double *dst = AB + (long long)c0 * g.ldab;
  for (long long e = threadIdx.x; e < tot; e += kThreads) dst[e] = blk[e];
  __syncthreads();
}

// Steps of panel p applied to block b (b > p): interchange, then the rank-1
// update, column by column of the block, one step after the other.
// s_l[k*kl + t-1] = multiplier l_{j+t, j} of column j = p*kNB + k; s_pk[k] = pivot
// offset; s_zp[k] != 0 for an exactly zero pivot (no interchange, no update).
__device__ void apply_panel(const Geo &g, double *blk, int b, int p, const double *s_l, const int *s_pk,
                            const int *s_zp) {
  const int c0 = b * kNB, nc = min(kNB, g.n - c0);
  const long long ldab = g.ldab;
  for (int k = 0; k < kNB; ++k) {
    const int j = p * kNB + k;
    if (j >= g.n) break;
    if (s_zp[k]) continue;  // uniform
    const int km = min(g.kl, g.n - 1 - j);
    const int pk = s_pk[k];
    if (pk != 0) {
      if (threadIdx.x < nc) {
        const int c = c0 + threadIdx.x;
        if (c <= j + g.kv) {  // beyond the reach of row j both entries are structural zeros
          double *x = blk + threadIdx.x * ldab + (g.kv + j - c);
          double *y = x + pk;
          const double t0 = *x;
          *x = *y;
          *y = t0;
        }
      }
      __syncthreads();
    }
    if (km > 0) {
      const int tot = km * nc;
      for (int e = threadIdx.x; e < tot; e += kThreads) {
        const int cc = e / km, t = 1 + (e - cc * km);
        const int c = c0 + cc;
        if (c > j + g.kv) continue;
        double *col = blk + cc * ldab + (g.kv + j - c);
        const double u = col[0];
        if (nz(u)) col[t] = fma(-s_l[k * g.kl + t - 1], u, col[t]);
      }
      __syncthreads();
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1) k_gbtrf_wide(int n, int kl, int ku, double *__restrict__ AB,
                                                              long long ldab, int *__restrict__ ipiv,
                                                              int *__restrict__ d_info, int *__restrict__ flags) {
  extern __shared__ double smem[];
  __shared__ KeyIdx s_red[kThreads / 32];
  __shared__ int s_pk[kNB], s_zp[kNB], s_ok, s_p;
  Geo g;
  g.n = n;
  g.kl = kl;
  g.ku = ku;
  g.kv = kl + ku;
  g.ldab = ldab;
  g.npan = (n + kNB - 1) / kNB;
  int *err = flags;
  int *panel_ready = flags + 2;
  int *block_ready = flags + 2 + g.npan;
  double *s_l = smem;                        // kNB * kl multipliers of the current panel
  double *blocks = smem + (size_t)kNB * kl;  // kMaxActive blocks of kNB * ldab
  const long long bsz = (long long)kNB * ldab;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (blockIdx.x == 0) {
    // ---------------- panel CTA ----------------
    int info = 0;
    double *cur = blocks, *nxt = blocks + bsz;
    load_block(g, AB, cur, 0, true);
    for (int p = 0; p < g.npan; ++p) {
      const int c0 = p * kNB, nc = min(kNB, n - c0);
      for (int k = 0; k < nc; ++k) {
        const int j = c0 + k;
        const int km = min(kl, n - 1 - j);
        double *col = cur + k * ldab + g.kv;  // col[t] = entry (j+t, j)
        KeyIdx best{0ull, LLONG_MAX};
        for (int t = threadIdx.x; t <= km; t += kThreads) best = better(best, KeyIdx{abs_key(col[t]), t});
        best = warp_reduce_keyidx(best);
        if (lane == 0) s_red[warp] = best;
        __syncthreads();
        if (warp == 0) {
          KeyIdx v = lane < kThreads / 32 ? s_red[lane] : KeyIdx{0ull, LLONG_MAX};
          v = warp_reduce_keyidx(v);
          if (lane == 0) s_p = (int)v.idx;
        }
        __syncthreads();
        const int pr = s_p;
        const double pv = col[pr];
        const bool zp = !nz(pv);
        if (threadIdx.x == 0) {
          ipiv[j] = j + pr + 1;
          s_pk[k] = pr;
          s_zp[k] = zp ? 1 : 0;
        }
        if (zp) {
          if (info == 0) info = j + 1;
          __syncthreads();
          continue;
        }
        if (pr != 0) {
          if (threadIdx.x < nc - k && threadIdx.x <= g.kv) {  // columns j .. block end, rows j and j+pr
            const int c = j + threadIdx.x;
            double *x = cur + (c - c0) * ldab + (g.kv + j - c);
            const double t0 = x[0];
            x[0] = x[pr];
            x[pr] = t0;
          }
          __syncthreads();
        }
        const double r = rcp_rn(pv);
        for (int t = 1 + threadIdx.x; t <= km; t += kThreads) col[t] *= r;
        __syncthreads();
        const int rest = min(nc - 1 - k, g.kv);
        if (rest > 0 && km > 0) {
          for (int e = threadIdx.x; e < km * rest; e += kThreads) {
            const int cc = e / km, t = 1 + (e - cc * km);
            const int c = j + 1 + cc;
            double *cj = cur + (c - c0) * ldab + (g.kv + j - c);
            const double u = cj[0];
            if (nz(u)) cj[t] = fma(-col[t], u, cj[t]);
          }
          __syncthreads();
        }
      }
      // publish panel p: the block to AB (U rows, multipliers, pivots already out)
      for (int e = threadIdx.x; e < kNB * kl; e += kThreads) {
        const int k = e / kl, t = 1 + (e - k * kl);
        s_l[e] = (k < nc && t <= min(kl, n - 1 - (c0 + k))) ? cur[k * ldab + g.kv + t] : 0.0;
      }
      store_block(g, AB, cur, p);
      cta_signal(panel_ready + p);
      if (p + 1 < g.npan) {
        const bool ho = handed_off(g, p + 1);
        if (ho && !cta_wait(block_ready + p + 1, err, &s_ok)) break;
        load_block(g, AB, nxt, p + 1, !ho);
        apply_panel(g, nxt, p + 1, p, s_l, s_pk, s_zp);
        double *tmp = cur;
        cur = nxt;
        nxt = tmp;
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) *d_info = ld_acquire(err) ? -BANDLU_ERR_TIMEOUT : info;
  } else {
    // ---------------- update CTAs ----------------
    const int G = gridDim.x - 1, u = blockIdx.x - 1;
    for (int p = 0; p + 2 < g.npan; ++p) {
      // owned blocks that panel p updates here: b in [p+2, b_last(p)], b = 2 + u (mod G)
      const int lo = p + 2, hi = b_last(g, p);
      int b0 = lo + ((u - (lo - 2)) % G + G) % G;
      if (b0 > hi) continue;
      if (!cta_wait(panel_ready + p, err, &s_ok)) break;
      // panel p's multipliers and pivots (written by the panel CTA before panel_ready[p])
      const int c0 = p * kNB, nc = min(kNB, n - c0);
      for (int e = threadIdx.x; e < kNB * kl; e += kThreads) {
        const int k = e / kl, t = 1 + (e - k * kl);
        s_l[e] = (k < nc && t <= min(kl, n - 1 - (c0 + k)))
                     ? __ldcg(AB + (long long)(c0 + k) * ldab + g.kv + t)
                     : 0.0;
      }
      if (threadIdx.x < kNB) {
        const int k = threadIdx.x;
        s_pk[k] = k < nc ? __ldcg(ipiv + c0 + k) - 1 - (c0 + k) : 0;
        s_zp[k] = k < nc ? (nz(__ldcg(AB + (long long)(c0 + k) * ldab + g.kv)) ? 0 : 1) : 1;
      }
      __syncthreads();
      for (int b = b0; b <= hi; b += G) {
        double *blk = blocks + (long long)((b - 2) / G % kMaxActive) * bsz;
        const int pf = p_first(g, b);
        if (p == pf) load_block(g, AB, blk, b, true);
        apply_panel(g, blk, b, p, s_l, s_pk, s_zp);
        if (p == b - 2) {
          store_block(g, AB, blk, b);
          cta_signal(block_ready + b);
        }
      }
      __syncthreads();
    }
  }
}

}  // namespace

// Launch conditions: every update CTA holds at most kMaxActive blocks at once
// and both roles fit in shared memory.  Returns BANDLU_ERR_UNSUPPORTED_SHAPE
// (a positive code never seen by callers) when the shape does not qualify.
int launch_gbtrf_wide(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t s,
                      bool *used) {
  *used = false;
  if (n < 3 * kNB || kl < 1) return BANDLU_OK;
  int dev = 0, sms = 0, coop = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (!coop || sms < 2) return BANDLU_OK;
  const long long kv = (long long)kl + ku;
  const size_t smem = ((size_t)kNB * kl + (size_t)kMaxActive * kNB * (size_t)ldab) * sizeof(double);
  if (smem > 200 * 1024) return BANDLU_OK;
  const int G = sms - 1;
  const long long span = (kv - 1) / kNB + 2;  // blocks one panel updates, at most
  if (span > (long long)kMaxActive * G) return BANDLU_OK;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(k_gbtrf_wide, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024) !=
        cudaSuccess)
      return BANDLU_ERR_CUDA;
    attr = true;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_gbtrf_wide, kThreads, smem) != cudaSuccess)
    return BANDLU_ERR_CUDA;
  if (per_sm < 1) return BANDLU_OK;
  // scratch: error flag, spare, panel_ready[npan], block_ready[npan]
  const long long npan = (n + kNB - 1) / kNB;
  const size_t fbytes = (size_t)(2 + 2 * npan) * sizeof(int);
  int *flags = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&flags), fbytes, s) != cudaSuccess) return BANDLU_ERR_CUDA;
  if (cudaMemsetAsync(flags, 0, fbytes, s) != cudaSuccess) return BANDLU_ERR_CUDA;
  int nn = (int)n, kkl = kl, kku = ku;
  long long lld = ldab;
  void *args[] = {&nn, &kkl, &kku, &AB, &lld, &ipiv, &d_info, &flags};
  const cudaError_t e = cudaLaunchCooperativeKernel((const void *)k_gbtrf_wide, dim3(sms), dim3(kThreads), args,
                                                    smem, s);
  cudaFreeAsync(flags, s);
  if (e != cudaSuccess) return BANDLU_ERR_CUDA;
  *used = true;
  return BANDLU_OK;
}

}  // namespace bandlu
