// peaks.cu -- microbenchmarks of the rates the rooflines are taken against
// (declared in include/bandlu_peaks.h): the FP64 FMA pipe, the FP64 tensor-core
// MMA (mma.sync .f64) and a read-only HBM stream.  The factorisation of
// Sec. III-A (Eq. S-N-N3) is FP64 arithmetic, the structure identification
// (Eq. IC-N2) one read of the dense matrix; these kernels measure what one
// GB300 delivers for each, so the benchmark's fractions use measured ceilings.
#include "bandlu_peaks.h"
#include "common.cuh"
#include "rcp.cuh"

namespace {

// Independent FMA chains per thread: the pipe sees `chains` instructions in
// flight per warp between dependent issues.
template <int C>
__global__ void k_peak_dfma(double *__restrict__ sink, int iters) {
  double a[C];
  const double b = 0.9999999999999, c = 1e-12 * (1 + (threadIdx.x & 7));
#pragma unroll
  for (int k = 0; k < C; ++k) a[k] = 1.0 + 1e-3 * (k + threadIdx.x);
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int k = 0; k < C; ++k) a[k] = fma(a[k], b, c);
  }
  double s = 0.0;
#pragma unroll
  for (int k = 0; k < C; ++k) s += a[k];
  // one value per block keeps every chain live without a reduction in the timed loop
  if (threadIdx.x == 0) sink[blockIdx.x] = s;
  else if (s == -1.0) sink[blockIdx.x] = s;  // never true: the chains stay observable
}

__device__ __forceinline__ void mma_m8n8k4(double &d0, double &d1, double a, double b) {
  asm volatile("mma.sync.aligned.m8n8k4.row.col.f64.f64.f64.f64 {%0, %1}, {%2}, {%3}, {%0, %1};"
               : "+d"(d0), "+d"(d1)
               : "d"(a), "d"(b));
}

__device__ __forceinline__ void mma_m16n8k16(double (&d)[4], const double (&a)[8], const double (&b)[4]) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f64.f64.f64.f64 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7, %8, %9, %10, %11}, {%12, %13, %14, %15}, {%0, %1, %2, %3};"
      : "+d"(d[0]), "+d"(d[1]), "+d"(d[2]), "+d"(d[3])
      : "d"(a[0]), "d"(a[1]), "d"(a[2]), "d"(a[3]), "d"(a[4]), "d"(a[5]), "d"(a[6]), "d"(a[7]), "d"(b[0]),
        "d"(b[1]), "d"(b[2]), "d"(b[3]));
}

template <int C>
__global__ void k_peak_dmma_m8n8k4(double *__restrict__ sink, int iters) {
  double d0[C], d1[C];
  const double a = 1e-3 * (1 + (threadIdx.x & 3)), b = 1e-3 * (1 + (threadIdx.x & 1));
#pragma unroll
  for (int k = 0; k < C; ++k) d0[k] = d1[k] = 0.0;
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int k = 0; k < C; ++k) mma_m8n8k4(d0[k], d1[k], a, b);
  }
  double s = 0.0;
#pragma unroll
  for (int k = 0; k < C; ++k) s += d0[k] + d1[k];
  if (threadIdx.x == 0) sink[blockIdx.x] = s;
  else if (s == -1.0) sink[blockIdx.x] = s;
}

template <int C>
__global__ void k_peak_dmma_m16n8k16(double *__restrict__ sink, int iters) {
  double d[C][4], a[8], b[4];
#pragma unroll
  for (int e = 0; e < 8; ++e) a[e] = 1e-3 * (1 + ((threadIdx.x + e) & 3));
#pragma unroll
  for (int e = 0; e < 4; ++e) b[e] = 1e-3 * (1 + ((threadIdx.x + e) & 1));
#pragma unroll
  for (int k = 0; k < C; ++k)
#pragma unroll
    for (int e = 0; e < 4; ++e) d[k][e] = 0.0;
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int k = 0; k < C; ++k) mma_m16n8k16(d[k], a, b);
  }
  double s = 0.0;
#pragma unroll
  for (int k = 0; k < C; ++k) s += d[k][0] + d[k][1] + d[k][2] + d[k][3];
  if (threadIdx.x == 0) sink[blockIdx.x] = s;
  else if (s == -1.0) sink[blockIdx.x] = s;
}

// Each block reads contiguous chunks of 512 x 4 16-byte vectors (32 KiB), chunk c
// by block c mod gridDim: every warp load is one contiguous 512-byte run.
__global__ void __launch_bounds__(512) k_peak_read(const ulonglong2 *__restrict__ p, long long nvec,
                                                   unsigned long long *__restrict__ sink) {
  constexpr int U = 4;
  __shared__ unsigned long long acc;
  if (threadIdx.x == 0) acc = 0ull;
  __syncthreads();
  unsigned long long x = 0ull;
  const long long chunk = (long long)blockDim.x * U;
  const long long nchunks = (nvec + chunk - 1) / chunk;
  for (long long c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const long long v0 = c * chunk + threadIdx.x;
    ulonglong2 a[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const long long v = v0 + (long long)u * blockDim.x;
      a[u] = v < nvec ? __ldcs(p + v) : make_ulonglong2(0ull, 0ull);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) x ^= a[u].x ^ a[u].y;
  }
  const unsigned lo = __reduce_xor_sync(bandlu::FULL, (unsigned)x),
                 hi = __reduce_xor_sync(bandlu::FULL, (unsigned)(x >> 32));
  if ((threadIdx.x & 31) == 0) atomicXor(&acc, ((unsigned long long)hi << 32) | lo);
  __syncthreads();
  if (threadIdx.x == 0) sink[blockIdx.x] = acc;
}

// One block; thread 0 times `iters` rounds of 16 instances of one operation.
template <int OP>
__global__ void k_peak_warp_costs(unsigned long long *__restrict__ clk, double *__restrict__ sink, int iters) {
  __shared__ __align__(16) double sm[32][32];
  const int t = threadIdx.x, lane = t & 31, w = t >> 5;
  double x = 1.0 + 1e-3 * lane, c8[8];
  unsigned u = 7u * lane + 3u;
#pragma unroll
  for (int k = 0; k < 8; ++k) c8[k] = x + k;
  sm[w][lane] = x;
  __syncthreads();
  const long long t0 = clock64();
  for (int it = 0; it < iters; ++it) {
    if constexpr (OP == 0) {
#pragma unroll
      for (int j = 0; j < 16; ++j) x = fma(x, 0.9999999999999, 1e-12);
    } else if constexpr (OP == 1) {
#pragma unroll
      for (int r = 0; r < 2; ++r)
#pragma unroll
        for (int k = 0; k < 8; ++k) c8[k] = fma(c8[k], 0.9999999999999, 1e-12);
    } else if constexpr (OP == 2) {
#pragma unroll
      for (int j = 0; j < 16; ++j) x = __shfl_sync(bandlu::FULL, x, (lane + 1) & 31);
    } else if constexpr (OP == 3) {
      unsigned a = 0u;
#pragma unroll
      for (int j = 0; j < 16; ++j) a += __shfl_sync(bandlu::FULL, u, (lane + j) & 31);
      u += a & 1u;
    } else if constexpr (OP == 4) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        sm[w][lane] = x;
        __syncwarp();
        x = ((volatile double *)sm[w])[(lane + 1) & 31];
        __syncwarp();
      }
    } else if constexpr (OP == 5) {
      // opaque to the compiler, which would otherwise fold the affine recurrence
#pragma unroll
      for (int j = 0; j < 16; ++j) asm volatile("mad.lo.u32 %0, %0, %1, %2;" : "+r"(u) : "r"(2654435761u), "r"(lane));
    } else if constexpr (OP == 6) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const unsigned m = __reduce_max_sync(bandlu::FULL, u);
        u += (__ballot_sync(bandlu::FULL, u == m) & 1u) + 1u;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        bool special;
        x = bandlu::rcp_rn_fast(x, &special);
      }
    }
  }
  const long long t1 = clock64();
  double s = x + (double)u;
#pragma unroll
  for (int k = 0; k < 8; ++k) s += c8[k];
  sink[t] = s;
  if (t == 0) *clk = (unsigned long long)(t1 - t0);
}

}  // namespace

extern "C" {

int bandlu_peak_dfma(double *d_sink, int blocks, int threads, int chains, int iters, cudaStream_t stream) {
  if (d_sink == nullptr) return -1;
  if (blocks < 1) return -2;
  if (threads < 32 || threads > 1024 || threads % 32 != 0) return -3;
  if (chains < 1 || chains > 8) return -4;
  if (iters < 1) return -5;
  switch (chains) {
    case 1: k_peak_dfma<1><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    case 2: k_peak_dfma<2><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    case 3: k_peak_dfma<3><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    case 4: k_peak_dfma<4><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    case 5: k_peak_dfma<5><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    case 6: k_peak_dfma<6><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    case 7: k_peak_dfma<7><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
    default: k_peak_dfma<8><<<blocks, threads, 0, stream>>>(d_sink, iters); break;
  }
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

int bandlu_peak_dmma(int shape, double *d_sink, int blocks, int warps, int chains, int iters, cudaStream_t stream) {
  if (shape != 0 && shape != 1) return -1;
  if (d_sink == nullptr) return -2;
  if (blocks < 1) return -3;
  if (warps < 1 || warps > 32) return -4;
  if (chains < 1 || chains > 4) return -5;
  if (iters < 1) return -6;
  const int t = 32 * warps;
  if (shape == 0) {
    switch (chains) {
      case 1: k_peak_dmma_m8n8k4<1><<<blocks, t, 0, stream>>>(d_sink, iters); break;
      case 2: k_peak_dmma_m8n8k4<2><<<blocks, t, 0, stream>>>(d_sink, iters); break;
      case 3: k_peak_dmma_m8n8k4<3><<<blocks, t, 0, stream>>>(d_sink, iters); break;
      default: k_peak_dmma_m8n8k4<4><<<blocks, t, 0, stream>>>(d_sink, iters); break;
    }
  } else {
    switch (chains) {
      case 1: k_peak_dmma_m16n8k16<1><<<blocks, t, 0, stream>>>(d_sink, iters); break;
      case 2: k_peak_dmma_m16n8k16<2><<<blocks, t, 0, stream>>>(d_sink, iters); break;
      case 3: k_peak_dmma_m16n8k16<3><<<blocks, t, 0, stream>>>(d_sink, iters); break;
      default: k_peak_dmma_m16n8k16<4><<<blocks, t, 0, stream>>>(d_sink, iters); break;
    }
  }
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

int bandlu_peak_hbm_read(const void *d_buf, int64_t bytes, unsigned long long *d_sink, int blocks,
                         cudaStream_t stream) {
  if (d_buf == nullptr || (reinterpret_cast<uintptr_t>(d_buf) & 15u) != 0) return -1;
  if (bytes < 16 || bytes % 16 != 0) return -2;
  if (d_sink == nullptr) return -3;
  if (blocks < 1) return -4;
  k_peak_read<<<blocks, 512, 0, stream>>>(static_cast<const ulonglong2 *>(d_buf), bytes / 16, d_sink);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

int bandlu_peak_warp_costs(int op, unsigned long long *d_clk, double *d_sink, int warps, int iters,
                           cudaStream_t stream) {
  if (op < 0 || op > 7) return -1;
  if (d_clk == nullptr) return -2;
  if (d_sink == nullptr) return -3;
  if (warps < 1 || warps > 32) return -4;
  if (iters < 1) return -5;
  const int t = 32 * warps;
  switch (op) {
    case 0: k_peak_warp_costs<0><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    case 1: k_peak_warp_costs<1><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    case 2: k_peak_warp_costs<2><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    case 3: k_peak_warp_costs<3><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    case 4: k_peak_warp_costs<4><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    case 5: k_peak_warp_costs<5><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    case 6: k_peak_warp_costs<6><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
    default: k_peak_warp_costs<7><<<1, t, 0, stream>>>(d_clk, d_sink, iters); break;
  }
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // extern "C"
