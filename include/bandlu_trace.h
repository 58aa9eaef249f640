/*
 * bandlu_trace.h -- timeline of the wide-band factorisation (a development build,
 * not part of the method).
 *
 * The wide-band factorisation's default kernel runs as thread-block clusters whose
 * CTAs wait on one another (the panel CTA and its streamers, Sec. III-A's DGBTRF
 * split over SMs), and no hardware counter capture is taken of it.  The library
 * built with BANDLU_TRACE defined (libbandlu_trace.so; bandlu.py loads it when
 * BANDLU_TRACE=1) records instead the GPU's global timer, in nanoseconds, at the
 * panel boundaries and waits of that kernel.  The production library records
 * nothing: bandlu_trace_capacity() returns 0 there and the other two calls
 * return BANDLU_ERR_CUDA.
 *
 * The record is 4 roles x capacity() entries x 16 slots of uint64 (0 = not
 * recorded), role-major.  Entry q is panel q for the panel CTA and its
 * streamers (the streamer entry of block b applying panel b-r is q = b-r), and
 * block b for the loader; a later call overwrites what an earlier one wrote.
 *   role 0, panel CTA:    0 panel start, 1 step 2's records sent, 2 panel done,
 *                         3 block q+1 usable (the wait is over); for column step
 *                         k = 0..3: 4+3k step start, 5+3k the step's barrier passed
 *                         (every warp has published), 6+3k its records sent
 *   roles 1, 2, streamers 1 and 2:
 *                         0 block in, 1 first records seen, 2 wait for the last
 *                         step's records begins, 3 last records seen, 4 band sent
 *   role 3, the last streamer's loader (entry = block):
 *                         0 wait for the update CTA's hand-over begins, 1 over
 * Panels beyond capacity() are not recorded.
 */
#ifndef BANDLU_TRACE_H
#define BANDLU_TRACE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Entries recorded per role: 8192 in the traced build, 0 in the production build. */
int bandlu_trace_capacity(void);

/* Copies the first `count` words of the record to the HOST array `host`
 * (count <= 4 * 16 * capacity()).  Synchronous.  Returns 0, -1 (host null),
 * -2 (count out of range) or BANDLU_ERR_CUDA (also in the production build). */
int bandlu_trace_read(uint64_t *host, int64_t count);

/* Zeroes the record.  Synchronous.  Returns 0 or BANDLU_ERR_CUDA. */
int bandlu_trace_clear(void);

#ifdef __cplusplus
}
#endif

#endif /* BANDLU_TRACE_H */
