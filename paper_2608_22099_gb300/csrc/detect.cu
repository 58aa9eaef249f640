// detect.cu -- structure identification (Sec. II-A step 1; I(N) ~ O(N^2), Eq. IC-N2).
//
// One HBM-bound pass over the n x n row-major matrix.  Work items are
// (row, segment) pairs; a segment is blockDim.x * U consecutive 16-byte vectors
// of one row, so every warp load is a contiguous 512-byte run.  Each thread
// keeps the largest i-j and j-i over the nonzeros it sees, the block folds them
// with warp max-reductions, and one thread per block folds the block result
// into the two outputs with atomicMax.  The nonzero test is integer-only
// ((bits << 1) != 0), so the FP64 pipe is never used.
//
// The outputs start at zero: a one-thread kernel clears them and at once lets
// the detection kernel launch behind it (programmatic dependent launch); the
// detection kernel reads the whole matrix and waits for that kernel to finish
// (griddepcontrol.wait) only before its atomics, so the reset costs no gap
// between launches.  Where the rows are contiguous (lda = 2*ceil(n/2) and A
// 16-byte aligned) the matrix is one run of 16-byte vectors and every block
// reads an equal share of it; otherwise work items are row segments.
#include "common.cuh"

namespace bandlu {
namespace {

__device__ __forceinline__ void block_fold(int lmax, int umax, int *d_kl, int *d_ku) {
  __shared__ int s_l[32], s_u[32];
  lmax = __reduce_max_sync(FULL, lmax);
  umax = __reduce_max_sync(FULL, umax);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) { s_l[w] = lmax; s_u[w] = umax; }
  __syncthreads();
  if (w == 0) {
    const int nw = blockDim.x >> 5;
    lmax = lane < nw ? s_l[lane] : 0;
    umax = lane < nw ? s_u[lane] : 0;
    lmax = __reduce_max_sync(FULL, lmax);
    umax = __reduce_max_sync(FULL, umax);
    if (lane == 0) {
      // the reset kernel (the prerequisite grid) has cleared the outputs by now
      asm volatile("griddepcontrol.wait;" ::: "memory");
      if (lmax > 0) atomicMax(d_kl, lmax);
      if (umax > 0) atomicMax(d_ku, umax);
    }
  }
}

// 16-byte path: A 16-byte aligned and lda even, so every row starts aligned.
// Vector v of row i holds columns 2v and 2v+1.  When n is odd, 2v+1 of the last
// vector is the first padding column (lda >= n+1 then): it is read, and ignored,
// on rows 0..n-2, but the last row reads its final column alone with an 8-byte
// load, so nothing past element (n-1)*lda + n-1 is ever read.
template <int U>
__global__ void __launch_bounds__(512) k_detect_vec(const double *__restrict__ A, long long n, long long lda,
                                                    long long nv, long long nseg, int *d_kl, int *d_ku) {
  const long long items = n * nseg;
  const long long seglen = (long long)blockDim.x * U;
  int lmax = 0, umax = 0;
  for (long long it = blockIdx.x; it < items; it += gridDim.x) {
    const long long i = it / nseg;
    const long long s = it - i * nseg;
    const ulonglong2 *row = reinterpret_cast<const ulonglong2 *>(A + i * lda);
    const long long v0 = s * seglen + threadIdx.x;
    // the vector that would reach past the matrix's last element
    const long long vcut = ((n & 1) && i == n - 1) ? nv - 1 : nv;
    ulonglong2 x[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const long long v = v0 + (long long)u * blockDim.x;
      if (v < vcut)
        x[u] = __ldcs(row + v);
      else if (v < nv)
        x[u] = make_ulonglong2(__ldcs(reinterpret_cast<const unsigned long long *>(row + v)), 0ull);
      else
        x[u] = make_ulonglong2(0ull, 0ull);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (((x[u].x << 1) | (x[u].y << 1)) != 0ull) {  // rare in a banded matrix
        const long long j0 = 2 * (v0 + (long long)u * blockDim.x);
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
  block_fold(lmax, umax, d_kl, d_ku);
}

// Contiguous rows (lda = 2*nv): vector f = i*nv + v of the flat run holds columns 2v
// and 2v+1 of row i and sits at A + 2f.  Block b reads vectors [b*chunk, (b+1)*chunk),
// chunk a multiple of 32.  When n is odd the second half of every row's last vector is
// the padding column; the matrix's very last vector is read as its first element alone.
template <int U>
__global__ void __launch_bounds__(512) k_detect_flat(const double *__restrict__ A, long long n, long long nv,
                                                     long long chunk, int *d_kl, int *d_ku) {
  const long long V = n * nv;
  const long long f0 = (long long)blockIdx.x * chunk;
  const long long f1 = min(V, f0 + chunk);
  const ulonglong2 *base = reinterpret_cast<const ulonglong2 *>(A);
  const long long vlast = (n & 1) ? V - 1 : V;  // vectors from here on would reach past the matrix
  const long long step = (long long)blockDim.x * U;
  int lmax = 0, umax = 0;
  for (long long f = f0 + threadIdx.x; f < f1; f += step) {
    ulonglong2 x[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const long long g = f + (long long)u * blockDim.x;
      if (g < min(f1, vlast))
        x[u] = __ldcs(base + g);
      else if (g < f1)
        x[u] = make_ulonglong2(__ldcs(reinterpret_cast<const unsigned long long *>(base + g)), 0ull);
      else
        x[u] = make_ulonglong2(0ull, 0ull);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (((x[u].x << 1) | (x[u].y << 1)) != 0ull) {  // rare in a banded matrix
        const long long g = f + (long long)u * blockDim.x;
        const long long i = g / nv;
        const long long j0 = 2 * (g - i * nv);
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
  block_fold(lmax, umax, d_kl, d_ku);
}

// Clears the outputs; the detection kernel behind it may start at once.
__global__ void k_detect_reset(int *d_kl, int *d_ku) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  *d_kl = 0;
  *d_ku = 0;
}

// Launch with programmatic stream serialisation: the kernel may begin while the
// reset kernel before it runs, and waits for it (griddepcontrol.wait) before writing.
template <typename... P, typename... Arg>
cudaError_t launch_after_reset(void (*k)(P...), unsigned grid, unsigned block, cudaStream_t s, Arg... a) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, static_cast<P>(a)...);
}

// 8-byte path for any alignment / odd lda.
__global__ void __launch_bounds__(256) k_detect_scalar(const double *__restrict__ A, long long n, long long lda,
                                                       long long nseg, int *d_kl, int *d_ku) {
  const long long items = n * nseg;
  int lmax = 0, umax = 0;
  for (long long it = blockIdx.x; it < items; it += gridDim.x) {
    const long long i = it / nseg;
    const long long s = it - i * nseg;
    const unsigned long long *row = reinterpret_cast<const unsigned long long *>(A + i * lda);
    const long long j0 = s * (long long)blockDim.x * 4 + threadIdx.x;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const long long j = j0 + (long long)u * blockDim.x;
      if (j < n && nz_bits(__ldcs(row + j))) {
        lmax = max(lmax, (int)(i - j));
        umax = max(umax, (int)(j - i));
      }
    }
  }
  block_fold(lmax, umax, d_kl, d_ku);
}

}  // namespace

int launch_detect(const double *A, int64_t n, int64_t lda, int *d_kl, int *d_ku, cudaStream_t s) {
  k_detect_reset<<<1, 1, 0, s>>>(d_kl, d_ku);
  BANDLU_CHECK_LAUNCH();
  if (n <= 1) return BANDLU_OK;
  const int sms = device_sms();
  const bool vec = ((reinterpret_cast<uintptr_t>(A) & 15u) == 0) && (lda % 2 == 0);
  cudaError_t e;
  if (vec) {
    const long long nv = (n + 1) / 2;
    if (lda == 2 * nv) {
      // one contiguous run of n*nv vectors, in equal chunks of whole warps
      const long long V = n * nv;
      const int B = V >= (1ll << 20) ? 512 : 256;
      const long long G0 = V >= (1ll << 20) ? (long long)sms * 4 : (long long)sms * 8;
      long long chunk = (V + G0 - 1) / G0;
      chunk = (chunk + 31) / 32 * 32;
      const long long grid = (V + chunk - 1) / chunk;
      e = V >= (1ll << 20) ? launch_after_reset(k_detect_flat<4>, (unsigned)grid, B, s, A, n, nv, chunk, d_kl, d_ku)
                           : launch_after_reset(k_detect_flat<2>, (unsigned)grid, B, s, A, n, nv, chunk, d_kl, d_ku);
    } else if (nv >= 2048) {
      const int B = 512;
      const long long nseg = (nv + (long long)B * 4 - 1) / ((long long)B * 4);
      const long long items = n * nseg;
      const long long grid = items < (long long)sms * 4 ? items : (long long)sms * 4;
      e = launch_after_reset(k_detect_vec<4>, (unsigned)grid, B, s, A, n, lda, nv, nseg, d_kl, d_ku);
    } else if (nv >= 512) {
      const int B = 128;
      const long long nseg = (nv + (long long)B * 4 - 1) / ((long long)B * 4);
      const long long items = n * nseg;
      const long long grid = items < (long long)sms * 16 ? items : (long long)sms * 16;
      e = launch_after_reset(k_detect_vec<4>, (unsigned)grid, B, s, A, n, lda, nv, nseg, d_kl, d_ku);
    } else {
      const int B = nv >= 128 ? 128 : 32;
      const long long nseg = (nv + B - 1) / B;
      const long long items = n * nseg;
      const long long grid = items < (long long)sms * 16 ? items : (long long)sms * 16;
      e = launch_after_reset(k_detect_vec<1>, (unsigned)grid, B, s, A, n, lda, nv, nseg, d_kl, d_ku);
    }
  } else {
    const int B = 256;
    const long long nseg = (n + (long long)B * 4 - 1) / ((long long)B * 4);
    const long long items = n * nseg;
    const long long grid = items < (long long)sms * 8 ? items : (long long)sms * 8;
    e = launch_after_reset(k_detect_scalar, (unsigned)grid, B, s, A, n, lda, nseg, d_kl, d_ku);
  }
  if (e != cudaSuccess) return BANDLU_ERR_CUDA;
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // namespace bandlu
