/*
 * bandlu_peaks.h -- hardware-rate microbenchmarks of libbandlu.so (not part of
 * the method).
 *
 * The factorisation of Sec. III-A (f(N) ~ O(N*P*Q), Eq. S-N-N3) is FP64
 * arithmetic and the structure identification (I(N) ~ O(N^2), Eq. IC-N2) is one
 * read of the dense matrix.  Their roofline fractions need the GPU's own FP64
 * and read-bandwidth ceilings, which the vendor's nominal figures do not give
 * reliably for this part.  These kernels measure them: the benchmark times each
 * launch with CUDA events on `stream` and divides the work stated below by the
 * time.
 *
 * Every function enqueues ONE kernel launch on `stream` and returns 0, a
 * negative -i for an invalid argument i (nothing launched), or
 * BANDLU_ERR_CUDA (1000).  All pointers are DEVICE pointers owned by the caller.
 * The kernels only read their input and write their sink; they never wait on
 * anything.
 */
#ifndef BANDLU_PEAKS_H
#define BANDLU_PEAKS_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* FP64 FMA rate.  blocks x threads threads each run `chains` independent chains
 * of `iters` dependent fma(a, b, c) (1 <= chains <= 8; threads a multiple of 32,
 * 32..1024; iters >= 1).  Work = 2 * blocks * threads * chains * iters flops.
 * d_sink: `blocks` doubles, one result per block (keeps the chains live). */
int bandlu_peak_dfma(double *d_sink, int blocks, int threads, int chains, int iters, cudaStream_t stream);

/* FP64 tensor-core (DMMA, mma.sync) rate.  shape 0: m8n8k4, shape 1: m16n8k16
 * (both .f64 inputs and accumulators).  Each warp of blocks x warps warps keeps
 * `chains` independent accumulators (1..4) and issues `iters` MMAs into each.
 * Work = 2*M*N*K * blocks * warps * chains * iters flops (M*N*K = 256 for shape 0,
 * 2048 for shape 1).  d_sink: `blocks` doubles. */
int bandlu_peak_dmma(int shape, double *d_sink, int blocks, int warps, int chains, int iters, cudaStream_t stream);

/* Read-only HBM stream: reads the `bytes` bytes at d_buf (16-byte aligned,
 * bytes a multiple of 16) once with streaming 16-byte loads, in contiguous
 * 32 KiB chunks dealt round-robin to `blocks` blocks of 512 threads.
 * Work = bytes read.  d_sink: `blocks` 64-bit words (an XOR of what was read). */
int bandlu_peak_hbm_read(const void *d_buf, int64_t bytes, unsigned long long *d_sink, int blocks,
                         cudaStream_t stream);

/* Per-warp cost of one operation, in SM clock cycles.  ONE block of `warps` warps
 * (1..32) runs `iters` (>= 1) rounds of 16 instances of operation `op`:
 *   0  dependent fma(a, b, c) in FP64 (each uses the previous result)
 *   1  independent FP64 fma (8 chains per thread, two rounds)
 *   2  dependent 64-bit warp shuffle of a double (__shfl_sync, source lane + 1)
 *   3  independent 32-bit warp shuffles
 *   4  shared-memory round trip: a store, __syncwarp, a load of a neighbour's value
 *   5  dependent 32-bit integer multiply-add
 *   6  dependent redux.sync max + ballot (the pivot search's reduction)
 *   7  dependent correctly rounded FP64 reciprocal (the library's integer-pipe
 *      reciprocal of Sec. III-A's multipliers, x -> 1/x)
 * d_clk: 1 word, thread 0's clock64 cycles over the rounds (cycles per operation
 * per warp = *d_clk / (16 * iters)); d_sink: 32 * warps doubles (keeps the
 * results live).  op outside 0..7 is argument 1. */
int bandlu_peak_warp_costs(int op, unsigned long long *d_clk, double *d_sink, int warps, int iters,
                           cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* BANDLU_PEAKS_H */
