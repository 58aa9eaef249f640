/*
 * bandlu_selftest.h -- self-test hooks of libbandlu.so (not part of the method).
 *
 * The pivot chain of gbtrf forms 1/pivot with an integer-pipe reciprocal that
 * must equal IEEE round-to-nearest division bit for bit (the multipliers are
 * a * (1/pivot), as DGBTF2 forms them; Sec. III-A names DGBTRF).  These hooks
 * expose that reciprocal so the test suite can check it against the host's and
 * the GPU's own division.  The back substitution of gbtrs divides by the
 * diagonal of U, known before the dividend; it uses a division built on that
 * reciprocal (Markstein's iteration), exposed here for the same check.
 */
#ifndef BANDLU_SELFTEST_H
#define BANDLU_SELFTEST_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* y[i] = reciprocal of x[i] for i < n, computed on the host with the library's
 * reciprocal.  x and y are HOST arrays of n doubles. */
void bandlu_selftest_rcp_host(const double *x, double *y, int64_t n);

/* y[i] = 1/x[i] on the device: the library's reciprocal (use_division == 0) or
 * the compiler's double division (use_division != 0), for comparison.  x and y
 * are DEVICE arrays of n doubles; asynchronous on `stream`.
 * Returns 0, -1 (x null), -2 (y null), -3 (n < 0) or BANDLU_ERR_CUDA. */
int bandlu_selftest_rcp_device(const double *x, double *y, int64_t n, int use_division, cudaStream_t stream);

/* q[i] = x[i] / d[i] for i < n with the library's known-divisor division, on
 * the host.  x, d and q are HOST arrays of n doubles. */
void bandlu_selftest_div_host(const double *x, const double *d, double *q, int64_t n);

/* The back substitution's quotient with its zero test, on the host: q[i] = x[i]
 * for a zero x[i] (either sign: no division, the sign kept), else x[i] / d[i]
 * with the known-divisor division.  x, d and q are HOST arrays of n doubles. */
void bandlu_selftest_div_nz_host(const double *x, const double *d, double *q, int64_t n);

/* q[i] = x[i] / d[i] on the device: the library's known-divisor division
 * (use_division == 0) or the compiler's double division (use_division != 0).
 * x, d and q are DEVICE arrays of n doubles; asynchronous on `stream`.
 * Returns 0, -1 (x null), -2 (d null), -3 (q null), -4 (n < 0) or BANDLU_ERR_CUDA. */
int bandlu_selftest_div_device(const double *x, const double *d, double *q, int64_t n, int use_division,
                               cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* BANDLU_SELFTEST_H */
