/*
 * bandlu.h -- C ABI of the GB300 (sm_103a) structure-aware banded LU library.
 *
 * The library implements the hot path of the structure-aware dispatch of
 * Lujan & Edelman, "When Structure is Silent: Opportunities for Algorithmic
 * Dispatch in Linear Algebra" (HPEC 2025), Sec. II-A (three steps: identify the
 * structure, convert the format, run the specialised algorithm) instantiated
 * for LU of banded matrices stored dense (Sec. III, Listing 2).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Dense input A: fp64, ROW-major, n x n, leading dimension lda >= max(1, n):
 *    element (i, j) is A[i*lda + j].  A is never modified.
 *  - Band storage AB: fp64, COLUMN-major, ldab x n, LAPACK xGBTRF layout
 *    (Sec. I-A cites xGBTRF): with kv = kl + ku, element (i, j) of the band
 *    lives at AB[(kv + i - j) + j*ldab]; rows 0..kl-1 are fill rows that row
 *    interchanges spill into; ldab >= 2*kl + ku + 1.
 *  - ipiv: int32, 1-based (LAPACK): row j was interchanged with row ipiv[j]-1.
 *  - All pointers are DEVICE pointers owned by the caller unless the name starts
 *    with h_ (host pointer).  Device buffers must not overlap.  The library
 *    keeps no pointer after a call returns.
 *  - Work is enqueued on `stream` (0 = legacy default stream) and runs
 *    asynchronously unless a function says otherwise.
 *  - Return value: BANDLU_OK, a negative number -i when argument i (1-based) is
 *    invalid (nothing is enqueued), or one of the positive codes below.  No
 *    entry point traps, asserts or hangs on the device.
 *  - Indexing is 64-bit throughout; n is limited to 2^31 - 1 and kl, ku to
 *    n - 1 (they are int32 in the outputs).  A leading dimension or stride
 *    whose extent over the matrix (or batch) does not fit a 64-bit offset is
 *    rejected like any other invalid argument.
 */
#ifndef BANDLU_H
#define BANDLU_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BANDLU_OK 0
/* dispatch_lu / dispatch_lu_batched: the dispatch predicate declined the band
 * path; nothing was factored (AB and ipiv untouched for that matrix). */
#define BANDLU_NOT_BANDED 1
/* a CUDA runtime call or kernel launch failed (cudaGetLastError is left set) */
#define BANDLU_ERR_CUDA 1000
/* a bounded device-side wait gave up; the results of the call are invalid */
#define BANDLU_ERR_TIMEOUT 1001
/* dispatch_lu_noalloc: the call would need more scratch than its static array holds */
#define BANDLU_ERR_SCRATCH 1002

/* Branches of the backslash dispatch (Listing 1, Sec. I-A), in the order it
 * tests them: bandlu_classify and dispatch_backslash report one of these. */
#define BANDLU_KIND_DIAGONAL 1 /* kl == 0 and ku == 0 (istril and istriu) */
#define BANDLU_KIND_LOWER 2    /* ku == 0: lower triangle of bandwidth kl (istril) */
#define BANDLU_KIND_UPPER 3    /* kl == 0: upper triangle of bandwidth ku (istriu) */
#define BANDLU_KIND_BANDED 4   /* LU through the band path: the dispatch predicate holds */
#define BANDLU_KIND_DENSE 5    /* LU the dense way: left to the caller */

/*
 * detect_bandwidth -- structure identification, step 1 of Sec. II-A; cost
 * I(N) ~ O(N^2) (Sec. III-A, Eq. IC-N2); banded_structure(A) in Listing 2.
 *
 * Inspects every element of A once and writes
 *   *d_kl = max(0, max{ i - j : A(i,j) != 0 }),  *d_ku = max(0, max{ j - i : A(i,j) != 0 })
 * to DEVICE memory.  "Nonzero" is the IEEE comparison a != 0.0: -0.0 counts as
 * zero; NaN, +-Inf and subnormal values count as nonzero.  An all-zero matrix
 * or n <= 1 gives (0, 0).  Columns lda-n..lda-1 (padding) are not read as part
 * of the matrix.
 * Arguments: 1 A, 2 n >= 0, 3 lda >= max(1,n), 4 d_kl (non-null), 5 d_ku (non-null).
 * Scratch: none.  Fastest when A is 16-byte aligned and lda is even.
 */
int detect_bandwidth(const double *A, int64_t n, int64_t lda, int *d_kl, int *d_ku, cudaStream_t stream);

/*
 * dense_to_band -- format conversion, step 2 of Sec. II-A; cost C(N)
 * (Sec. III-A, Eq. IC-N2); BandedMatrix(A) in Listing 2.
 *
 * Writes all ldab x n entries of AB: AB(kv+i-j, j) = A(i,j) for
 * max(0, j-ku) <= i <= min(n-1, j+kl), and +0.0 everywhere else (fill rows,
 * the corner triangles and any rows beyond 2*kl+ku).  Entries of A outside the
 * band are not read.
 * Arguments: 1 A, 2 lda >= max(1,n), 3 n >= 0, 4 kl >= 0, 5 ku >= 0, 6 AB,
 * 7 ldab >= 2*kl+ku+1.  kl and ku must be less than n when n > 0.
 */
int dense_to_band(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                  cudaStream_t stream);

/*
 * gbtrf -- banded LU with partial pivoting, step 3 of Sec. II-A; cost
 * f(N) ~ O(N*P*Q) (Sec. III-A, Eq. S-N-N3); DGBTRF in Listing 2.
 *
 * Factors the band in AB in place as A = P_0 L_0 P_1 L_1 ... P_{n-1} L_{n-1} U
 * with LAPACK xGBTRF semantics: the pivot of column j is the FIRST entry of
 * largest magnitude among rows j..min(n-1, j+kl); the interchange is applied to
 * the columns of U; the multipliers l = a * (1/pivot) (a reciprocal, then one
 * multiply) of column j are stored in AB rows kv+1..kv+kl of column j, not
 * permuted by later interchanges; the trailing update is a = fma(-l, u, a) and
 * is skipped for a column whose pivot-row entry u is exactly zero.  U occupies
 * rows 0..kv.  The fill rows 0..kl-1 need not be zero on entry.
 * On exit *d_info (DEVICE) is 0, or j+1 for the first column j whose pivot is
 * exactly zero (that column is left unscaled and elimination continues, as
 * LAPACK does; this is not an error return).
 * Arguments: 1 n >= 0, 2 kl >= 0, 3 ku >= 0, 4 AB, 5 ldab >= 2*kl+ku+1,
 * 6 ipiv (n int32, device), 7 d_info (device).
 * Pivot comparisons follow the running-maximum order of LAPACK's IDAMAX: the
 * running best starts at the first candidate (row j) and a later candidate
 * replaces it only when its modulus is strictly larger.  So ties go to the
 * lowest row, and a NaN becomes the pivot only when it is the first candidate
 * (no later modulus compares larger than a NaN); a NaN below row j is never
 * chosen over an earlier candidate.
 * Scratch: for bands wide enough for the multi-CTA kernel, 8 + 8*ceil(n/4)
 * bytes of hand-off flags from the stream-ordered allocator (cudaMallocAsync
 * on `stream`, freed in stream order); otherwise none.
 */
int gbtrf(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t stream);

/*
 * detect_bandwidth_cm, dense_to_band_cm -- detect_bandwidth and dense_to_band
 * for a COLUMN-major A (the layout of the Julia code the paper's listings are
 * written in): element (i, j) is A[i + j*lda].  Same definitions, arguments,
 * outputs and return codes as the row-major calls; A's columns are contiguous,
 * so the conversion reads each band column in one run.
 */
int detect_bandwidth_cm(const double *A, int64_t n, int64_t lda, int *d_kl, int *d_ku, cudaStream_t stream);
int dense_to_band_cm(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                     cudaStream_t stream);

/*
 * dispatch_lu -- the whole strategy of Sec. II-A for one matrix
 * (structure_aware_lu of Listing 2 without the dense branch).
 *
 * Runs detect_bandwidth, reads (kl, ku) back to the host (the call waits for
 * `stream` once), applies the dispatch predicate, and if it holds runs
 * dense_to_band and gbtrf on `stream` (those two stay asynchronous).
 * The predicate is the speedup constraint of Eq. su-con (Sec. II-B),
 * I(N) + C(N) + f(N) < F(N), with the operation counts I = n^2,
 * C = n*(kl+ku+1), f = n*kl*(2*(kl+ku)+1) (worst-case fill) and F = 2n^3/3,
 * evaluated exactly in integers, together with the capacity check
 * 2*kl+ku+1 <= ldab.
 * Returns BANDLU_OK (band path enqueued; *d_info is written by gbtrf) or
 * BANDLU_NOT_BANDED (nothing further enqueued; AB, ipiv, d_info untouched).
 * *h_kl and *h_ku (HOST) receive the detected bandwidths in both cases.
 * Arguments: 1 A, 2 n, 3 lda, 4 AB, 5 ldab >= 1, 6 ipiv, 7 h_kl, 8 h_ku, 9 d_info.
 * Scratch: 8 bytes of device memory for the detected bandwidths, taken from the
 * stream-ordered allocator (cudaMallocAsync) and released before returning.
 */
int dispatch_lu(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *h_kl,
                int *h_ku, int *d_info, cudaStream_t stream);

/*
 * dispatch_lu_cm -- dispatch_lu for a COLUMN-major A (A(i,j) = A[i + j*lda]):
 * detect_bandwidth_cm, the same predicate, dense_to_band_cm and gbtrf.  Same
 * arguments, outputs, return codes and scratch as dispatch_lu.
 */
int dispatch_lu_cm(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *h_kl,
                   int *h_ku, int *d_info, cudaStream_t stream);

/*
 * dispatch_lu_async -- dispatch_lu with the decision taken on the device: the
 * same identification, predicate, conversion and factorisation, enqueued on
 * `stream` without any host synchronisation or allocation, so that a caller can
 * queue dispatches back to back or capture the call in a CUDA graph.
 * Outputs, all in DEVICE memory: *d_kl, *d_ku (as detect_bandwidth), *d_status
 * (BANDLU_OK: factored, *d_info written by the factorisation; BANDLU_NOT_BANDED:
 * declined, AB, ipiv and *d_info untouched).  The factors are those of
 * dispatch_lu (the same kernels and order of operations) for every band whose
 * active window fits a shared-memory window of one CTA (kl <= 27 and
 * 2*kl+ku+1 <= 256); wider bands are factored by a single CTA column by column
 * (the same results, more slowly: the multi-CTA kernel dispatch_lu uses there
 * is sized from kl on the host).
 * Arguments: 1 A, 2 n, 3 lda, 4 AB, 5 ldab (1 <= ldab < 2^31), 6 ipiv,
 * 7 d_kl, 8 d_ku, 9 d_status, 10 d_info (DEVICE, distinct).
 * Returns BANDLU_OK (work enqueued), -i for a bad argument i, BANDLU_ERR_CUDA.
 * Scratch: none.
 */
int dispatch_lu_async(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *d_kl,
                      int *d_ku, int *d_status, int *d_info, cudaStream_t stream);

/*
 * gbtrs -- the solve after the factorisation: the backslash operator the
 * dispatch of Listing 1 (Sec. I-A) stands for, on the band path (LAPACK xGBTRS,
 * no transpose).  Solves A X = B with A = P0 L0 P1 L1 ... U as left in AB and
 * ipiv by gbtrf (same kl, ku, ldab).
 *   forward, j = 0..n-2 (kl > 0): rows j and ipiv[j]-1 of B are interchanged;
 *     then, where b = B(j, c) != 0, B(j+t, c) = fma(-l_{j+t,j}, b, B(j+t, c)) for
 *     t = 1..min(kl, n-1-j);
 *   backward, j = n-1..0: where B(j, c) != 0, B(j, c) = B(j, c) / U(j,j) and
 *     B(i, c) = fma(-B(j, c), U(i,j), B(i, c)) for i = max(0, j-kl-ku)..j-1.
 * (The zero tests are those of the reference BLAS.)  A singular U (a zero
 * U(j,j)) yields infinities or NaNs, as in LAPACK; callers check info first.
 * Arguments (all DEVICE pointers): 1 n >= 0, 2 kl >= 0, 3 ku >= 0, 4 nrhs >= 0,
 * 5 AB (read only), 6 ldab >= 2*kl+ku+1, 7 ipiv (1-based, read only),
 * 8 B (COLUMN-major n x nrhs, overwritten with X), 9 ldb >= max(1, n).
 * Returns BANDLU_OK, -i for a bad argument i, BANDLU_ERR_CUDA.  Asynchronous.
 */
int gbtrs(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
          int64_t ldb, cudaStream_t stream);

/*
 * dispatch_solve -- A X = B through the structure-aware dispatch: dispatch_lu,
 * then, on the band path, gbtrs with the factors it produced (the backslash of
 * Listing 1 with the dense branch left to the caller).
 * Returns what dispatch_lu returns.  On BANDLU_OK the solve is enqueued on
 * `stream`; it reads *d_info on the device and leaves B as it is when the
 * factor is singular (info > 0), so no further host synchronisation is needed.
 * On BANDLU_NOT_BANDED nothing further is enqueued and B is untouched.
 * Arguments: 1 A, 2 n, 3 lda, 4 B (COLUMN-major n x nrhs), 5 ldb >= max(1, n),
 * 6 nrhs >= 0, 7 AB, 8 ldab >= 1, 9 ipiv, 10 h_kl, 11 h_ku (HOST), 12 d_info.
 * Scratch: as dispatch_lu.
 */
int dispatch_solve(const double *A, int64_t n, int64_t lda, double *B, int64_t ldb, int64_t nrhs, double *AB,
                   int64_t ldab, int *ipiv, int *h_kl, int *h_ku, int *d_info, cudaStream_t stream);

/*
 * trsv_band -- the LowerTriangular / UpperTriangular solve of the backslash
 * dispatch (Listing 1, Sec. I-A), on a triangle of bandwidth k read in place
 * from the dense ROW-major A (no format conversion; only the band is read).
 * xTRTRS semantics: *d_info = the first i (1-based) with A(i,i) == 0 and then B
 * is left as it is, else 0 and every column b of B is overwritten with the
 * solution by the column-oriented substitution of the reference BLAS (xTBSV, no
 * transpose), with its zero test and one fma per elimination:
 *   lower, j = 0..n-1:  if b_j != 0:  b_j = b_j / A(j,j);  b_i = fma(-b_j, A(i,j), b_i), i = j+1..min(n-1, j+k)
 *   upper, j = n-1..0:  if b_j != 0:  b_j = b_j / A(j,j);  b_i = fma(-b_j, A(i,j), b_i), i = max(0, j-k)..j-1
 * Arguments: 1 lower (1 = lower, 0 = upper triangle), 2 n >= 0, 3 k (0 <= k <=
 * max(0, n-1)), 4 A, 5 lda >= max(1, n), 6 B (COLUMN-major n x nrhs, DEVICE),
 * 7 ldb >= max(1, n), 8 nrhs >= 0, 9 d_info (DEVICE, always written).
 * Returns BANDLU_OK, -i for a bad argument i, BANDLU_ERR_CUDA.  Asynchronous.
 * Scratch: none.
 */
int trsv_band(int lower, int64_t n, int k, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs,
              int *d_info, cudaStream_t stream);

/*
 * diag_solve -- the Diagonal solve of the backslash dispatch (Listing 1): B(i,c)
 * = B(i,c) / A(i,i) (IEEE division), with A dense ROW-major and only its
 * diagonal read.  *d_info = the first i (1-based) with A(i,i) == 0 (then B is
 * left as it is), else 0.
 * Arguments: 1 n >= 0, 2 A, 3 lda >= max(1, n), 4 B (COLUMN-major n x nrhs),
 * 5 ldb >= max(1, n), 6 nrhs >= 0, 7 d_info (DEVICE, always written).
 * Returns BANDLU_OK, -i for a bad argument i, BANDLU_ERR_CUDA.  Asynchronous.
 */
int diag_solve(int64_t n, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs, int *d_info,
               cudaStream_t stream);

/*
 * bandlu_classify -- the branch Listing 1 takes for detected bandwidths (kl, ku)
 * (host only, no GPU work): BANDLU_KIND_DIAGONAL when kl == ku == 0, LOWER when
 * ku == 0, UPPER when kl == 0, otherwise BANDED when the dispatch predicate of
 * dispatch_lu holds for capacity ldab and DENSE when it does not.  Returns -1
 * for n < 0, kl < 0 or ku < 0.
 */
int bandlu_classify(int64_t n, int kl, int ku, int64_t ldab);

/*
 * dispatch_backslash -- A X = B through the backslash dispatch of Listing 1
 * (Sec. I-A) with the band path of Sec. II-A: detect_bandwidth, (kl, ku) read
 * back to the host (the call waits for `stream` once), bandlu_classify, then
 * the branch's solve enqueued on `stream`:
 *   DIAGONAL: diag_solve;  LOWER: trsv_band(1, n, kl);  UPPER: trsv_band(0, n, ku);
 *   BANDED: dense_to_band, gbtrf and gbtrs with AB and ipiv (the solve is
 *           skipped on the device when the factor is singular, as in dispatch_solve);
 *   DENSE: nothing is enqueued and B is untouched (the caller's dense LU).
 * *d_info is written by every branch but DENSE (first zero diagonal entry, or
 * gbtrf's info).  *h_kl, *h_ku and *h_kind (HOST) are always written.
 * Returns BANDLU_OK, BANDLU_NOT_BANDED (the DENSE branch), -i for a bad
 * argument i, or an error code.
 * Arguments: 1 A, 2 n, 3 lda, 4 B (COLUMN-major n x nrhs), 5 ldb >= max(1, n),
 * 6 nrhs >= 0, 7 AB, 8 ldab >= 1, 9 ipiv, 10 h_kl, 11 h_ku, 12 h_kind (HOST),
 * 13 d_info.  AB and ipiv are only written by the BANDED branch.
 * Scratch: as dispatch_lu.
 */
int dispatch_backslash(const double *A, int64_t n, int64_t lda, double *B, int64_t ldb, int64_t nrhs, double *AB,
                       int64_t ldab, int *ipiv, int *h_kl, int *h_ku, int *h_kind, int *d_info, cudaStream_t stream);

/*
 * dispatch_lu_batched -- the strategy of Sec. II-A applied to `batch`
 * independent n x n matrices in one call, with no host round trip.
 *
 * Matrix b is read from A + b*strideA (leading dimension lda); its band goes to
 * AB + b*strideAB (leading dimension ldab), its pivots to ipiv + b*strideP.
 * Every matrix gets its own (kl, ku) and its own predicate decision (as in
 * dispatch_lu, with the shared capacity ldab); per-matrix results go to the
 * DEVICE arrays d_kl[b], d_ku[b], d_info[b] and d_status[b] (BANDLU_OK or
 * BANDLU_NOT_BANDED; a declined matrix's AB and ipiv are untouched and its
 * d_info is 0).
 * Arguments: 1 A, 2 n, 3 lda, 4 strideA >= n*lda, 5 batch >= 0, 6 AB,
 * 7 ldab >= 1, 8 strideAB >= n*ldab, 9 ipiv, 10 strideP >= n, 11 d_kl, 12 d_ku,
 * 13 d_info, 14 d_status.
 * Scratch: none.
 */
int dispatch_lu_batched(const double *A, int64_t n, int64_t lda, int64_t strideA, int64_t batch, double *AB,
                        int64_t ldab, int64_t strideAB, int *ipiv, int64_t strideP, int *d_kl, int *d_ku,
                        int *d_info, int *d_status, cudaStream_t stream);

/*
 * dispatch_lu_noalloc -- dispatch_lu for callers that cannot allocate device
 * memory.  The paper has no counterpart: this is a deployment variant.
 *
 * dispatch_lu takes its 8 bytes of scratch (the detected kl, ku) from the
 * stream-ordered allocator on every call.  Some callers cannot let a library
 * allocate: a process whose device memory is entirely reserved by its own
 * caching allocator (an extra allocation can fail or fragment its pool), or a
 * latency-critical loop whose rules forbid allocation calls, which can take
 * driver locks or synchronize.  This entry point computes exactly what
 * dispatch_lu computes, with the same arguments, return codes and outputs, and
 * calls no cudaMalloc, cudaMallocAsync, cudaFree or other allocating routine.
 *
 * Scratch: a file-scope __device__ array of 256 bytes, of which one call uses
 * 8 (kl, ku), whatever n is; a call needing more returns BANDLU_ERR_SCRATCH.
 * Every GPU that loads the library holds the array until the process exits.
 * The first call on each device resolves the array's device address
 * (cudaGetSymbolAddress) with that device current, and keeps it for that
 * device's context; after a cudaDeviceReset the next call resolves it again in
 * the new context.  Make the first call on a device (and the first after a
 * reset) before any stream capture begins.  Like dispatch_lu, the call
 * synchronizes `stream` once to read the detected bandwidths.  All calls share
 * the one array and it keeps the last call's contents (each call clears the pair
 * before detecting), so calls whose work overlaps on the GPU (different streams
 * or threads, no ordering between them) race on it: serialise them.
 * Arguments: as dispatch_lu.
 */
int dispatch_lu_noalloc(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *h_kl,
                        int *h_ku, int *d_info, cudaStream_t stream);

/* Version string of the library build (host, static storage). */
const char *bandlu_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BANDLU_H */
