// convert.cu -- format conversion (Sec. II-A step 2; C(N), Eq. IC-N2).
//
// Dense row-major A -> LAPACK band storage AB (column-major, ldab x n).  A block
// owns T consecutive output columns [j0, j0+T), i.e. the contiguous run
// AB[j0*ldab, (j0+T)*ldab).  It zeroes a T x ldab shared-memory tile laid out
// exactly like that run, gathers the band part of rows j0-ku .. j0+T-1+kl of A
// into it (each row's band segment is contiguous in A, so a warp reads it with
// consecutive addresses), and streams the tile out with consecutive stores.
// Only band entries of A are read; every AB entry is written.  The gather is
// issued as 8-byte cp.async copies, so a warp has all its rows in flight at once
// instead of one load-store round trip per row; the zero fill touches only the
// tile positions the gather does not write (fill rows, band rows outside the
// matrix), so the two never meet.
#include "common.cuh"

namespace bandlu {
namespace {

// Fills the shared tile of output columns [j0, j0+tcols) (tile[c*ldab + r] = AB(r, j0+c))
// and returns after the block's barrier that makes it complete.
__device__ __forceinline__ void fill_band_tile(const double *__restrict__ A, long long lda, long long n, long long kl,
                                               long long ku, long long j0, int tcols, long long ldab, double *tile) {
  const long long kv = kl + ku;
  const int L = (int)ldab;
  const int tsize = tcols * L;
  for (int e = threadIdx.x; e < tsize; e += blockDim.x) {
    const int c = e / L, r = e - c * L;
    const long long i = j0 + c - kv + r;
    if (r < kl || r > kv + kl || i < 0 || i >= n) tile[e] = 0.0;
  }
  const long long i_lo = max(0ll, j0 - ku);
  const long long i_hi = min(n - 1, j0 + tcols - 1 + kl);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
  for (long long i = i_lo + warp; i <= i_hi; i += nwarps) {
    const long long c_lo = max(j0, i - kl);
    const long long c_hi = min(min(j0 + tcols - 1, i + ku), n - 1);
    for (long long c = c_lo + lane; c <= c_hi; c += 32) {
      const unsigned dst = (unsigned)__cvta_generic_to_shared(tile + (c - j0) * ldab + (kv + i - c));
      asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(dst), "l"(A + i * lda + c) : "memory");
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();
}

__global__ void __launch_bounds__(256) k_dense_to_band_tiled(const double *__restrict__ A, long long lda, long long n,
                                                             int kl, int ku, double *__restrict__ AB, long long ldab,
                                                             int T) {
  extern __shared__ double tile[];  // T * ldab, tile[c*ldab + r] = AB(r, j0+c)
  const long long j0 = (long long)blockIdx.x * T;
  const int tcols = (int)min((long long)T, n - j0);
  const long long tsize = (long long)tcols * ldab;
  fill_band_tile(A, lda, n, kl, ku, j0, tcols, ldab, tile);
  double *out = AB + j0 * ldab;
  for (long long e = threadIdx.x; e < tsize; e += blockDim.x) out[e] = tile[e];
}

// Direct form for very tall band storage: one thread per AB entry, consecutive
// threads on consecutive AB rows (coalesced stores; reads of A are strided).
__global__ void __launch_bounds__(256) k_dense_to_band_direct(const double *__restrict__ A, long long lda, long long n,
                                                              int kl, int ku, double *__restrict__ AB, long long ldab) {
  const long long kv = (long long)kl + ku;
  const long long total = n * ldab;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const long long j = e / ldab;
    const long long r = e - j * ldab;
    const long long i = j - kv + r;
    double v = 0.0;
    if (r >= kl && r <= kv + kl && i >= 0 && i < n) v = A[i * lda + j];
    AB[e] = v;
  }
}

// dispatch_lu_async: the decision taken on the device.  Every block reads the
// detected (kl, ku), applies the dispatch predicate (block 0 records it in
// *d_status) and, for a banded matrix, converts its tile as k_dense_to_band_tiled
// does (the tile size depends on ldab only).
__global__ void __launch_bounds__(256) k_decide_convert_tiled(const double *__restrict__ A, long long lda, long long n,
                                                              const int *__restrict__ d_kl,
                                                              const int *__restrict__ d_ku, int *__restrict__ d_status,
                                                              double *__restrict__ AB, long long ldab, int T) {
  const long long kl = *d_kl, ku = *d_ku;
  const bool banded = predicate_banded(n, kl, ku, ldab);
  if (blockIdx.x == 0 && threadIdx.x == 0) *d_status = banded ? BANDLU_OK : BANDLU_NOT_BANDED;
  if (!banded) return;  // whole block
  extern __shared__ double tile[];
  const long long j0 = (long long)blockIdx.x * T;
  const int tcols = (int)min((long long)T, n - j0);
  const long long tsize = (long long)tcols * ldab;
  fill_band_tile(A, lda, n, kl, ku, j0, tcols, ldab, tile);
  double *out = AB + j0 * ldab;
  for (long long e = threadIdx.x; e < tsize; e += blockDim.x) out[e] = tile[e];
}

// The direct form of the same, for very tall band storage.
__global__ void __launch_bounds__(256) k_decide_convert_direct(const double *__restrict__ A, long long lda,
                                                               long long n, const int *__restrict__ d_kl,
                                                               const int *__restrict__ d_ku,
                                                               int *__restrict__ d_status, double *__restrict__ AB,
                                                               long long ldab) {
  const long long kl = *d_kl, ku = *d_ku;
  const bool banded = predicate_banded(n, kl, ku, ldab);
  if (blockIdx.x == 0 && threadIdx.x == 0) *d_status = banded ? BANDLU_OK : BANDLU_NOT_BANDED;
  if (!banded) return;
  const long long kv = kl + ku;
  const long long total = n * ldab;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const long long j = e / ldab;
    const long long r = e - j * ldab;
    const long long i = j - kv + r;
    double v = 0.0;
    if (r >= kl && r <= kv + kl && i >= 0 && i < n) v = A[i * lda + j];
    AB[e] = v;
  }
}

// Column-major input, A(i,j) = A[i + j*lda]: one thread per AB entry; AB
// column j is A's column j shifted by kv - j, so consecutive threads read and
// write consecutive addresses.
__global__ void __launch_bounds__(256) k_dense_to_band_cm(const double *__restrict__ A, long long lda, long long n,
                                                          int kl, int ku, double *__restrict__ AB, long long ldab) {
  const long long kv = (long long)kl + ku;
  const long long total = n * ldab;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const long long j = e / ldab;
    const long long r = e - j * ldab;
    const long long i = j - kv + r;
    double v = 0.0;
    if (r >= kl && r <= kv + kl && i >= 0 && i < n) v = A[i + j * lda];
    AB[e] = v;
  }
}

constexpr int kTileSmemMax = 96 * 1024;

// Columns per tile for band storage of height ldab: enough blocks to cover the
// SMs for small n, at most 32; 0 when one column does not fit the tile.
int tile_columns(long long n, long long ldab) {
  const long long per_col = ldab * (long long)sizeof(double);
  if (per_col > kTileSmemMax) return 0;
  int T = (int)min(32ll, (long long)kTileSmemMax / per_col);
  while (T > 1 && (n + T - 1) / T < 304) T >>= 1;
  return T < 1 ? 1 : T;
}

}  // namespace

int launch_dense_to_band(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                         cudaStream_t s) {
  if (n == 0) return BANDLU_OK;
  const long long per_col = ldab * (long long)sizeof(double);
  const int T = tile_columns(n, ldab);
  if (T > 0) {
    const size_t smem = (size_t)T * per_col;
    if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_dense_to_band_tiled), kTileSmemMax)) return BANDLU_ERR_CUDA;
    const long long blocks = (n + T - 1) / T;
    k_dense_to_band_tiled<<<(unsigned)blocks, 256, smem, s>>>(A, lda, n, kl, ku, AB, ldab, T);
  } else {
    const long long total = n * ldab;
    long long blocks = (total + 255) / 256;
    if (blocks > 152ll * 32) blocks = 152ll * 32;
    k_dense_to_band_direct<<<(unsigned)blocks, 256, 0, s>>>(A, lda, n, kl, ku, AB, ldab);
  }
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

int launch_decide_convert(const double *A, int64_t lda, int64_t n, int64_t ldab, const int *d_kl, const int *d_ku,
                          int *d_status, double *AB, cudaStream_t s) {
  const int T = n > 0 ? tile_columns(n, ldab) : 0;  // n == 0: the direct kernel records the decision
  if (T > 0) {
    const size_t smem = (size_t)T * ldab * sizeof(double);
    if (!allow_dynamic_smem(reinterpret_cast<const void *>(k_decide_convert_tiled), kTileSmemMax))
      return BANDLU_ERR_CUDA;
    k_decide_convert_tiled<<<(unsigned)((n + T - 1) / T), 256, smem, s>>>(A, lda, n, d_kl, d_ku, d_status, AB, ldab,
                                                                          T);
  } else {
    long long blocks = (n * ldab + 255) / 256;
    if (blocks > 152ll * 32) blocks = 152ll * 32;
    if (blocks < 1) blocks = 1;
    k_decide_convert_direct<<<(unsigned)blocks, 256, 0, s>>>(A, lda, n, d_kl, d_ku, d_status, AB, ldab);
  }
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

int launch_dense_to_band_cm(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                            cudaStream_t s) {
  if (n == 0) return BANDLU_OK;
  long long blocks = (n * ldab + 255) / 256;
  if (blocks > 152ll * 64) blocks = 152ll * 64;
  k_dense_to_band_cm<<<(unsigned)blocks, 256, 0, s>>>(A, lda, n, kl, ku, AB, ldab);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu
