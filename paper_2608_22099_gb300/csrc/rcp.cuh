// rcp.cuh -- correctly rounded double reciprocal on the integer and FP32 pipes.
//
// GB300's FP64 pipe issues one warp instruction per 64 clocks per SMSP, so the
// ~7 dependent FP64 operations of a double division sit squarely on the pivot
// chain of the band LU.  This reciprocal uses integer arithmetic instead.  For a
// normal b = +-m * 2^(E-1075) with 2^52 <= m < 2^53 (E the biased exponent),
//   1/b = (2^105 / m) * 2^(970-E),
// so the rounded significand is q = Q + [2R > m] where Q = floor(2^105/m) and
// R = 2^105 - Q*m (no ties are possible: 2^106/m is not an integer for m > 2^52).
// Q is found as a quotient by approximate reciprocal with remainder correction
// (Knuth, TAOCP Vol. 2, Sec. 4.3.1): a Newton step on a two-float (double-float)
// representation of m gives Q within 2^9; one correction Q += (2^105 - Q*m)/m,
// the remainder's high bits times y's 24-bit significand in one integer
// multiply, brings Q within one unit; the exact remainder then fixes Q and
// decides the rounding.
// The result is the IEEE round-to-nearest 1/b, bit for bit.  Zeros, subnormals,
// infinities, NaN and |b| >= 2^1021 (whose reciprocal is subnormal) go to the
// ordinary division.
#pragma once

#include <cmath>
#include <cstdint>
#include <cstring>

namespace bandlu {

__host__ __device__ __forceinline__ float rcp_approx_f32(float x) {
#ifdef __CUDA_ARCH__
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
#else
  return 1.0f / x;
#endif
}

__host__ __device__ __forceinline__ uint64_t dbits(double x) {
#ifdef __CUDA_ARCH__
  return (uint64_t)__double_as_longlong(x);
#else
  uint64_t u;
  std::memcpy(&u, &x, 8);
  return u;
#endif
}

__host__ __device__ __forceinline__ double bitsd(uint64_t u) {
#ifdef __CUDA_ARCH__
  return __longlong_as_double((long long)u);
#else
  double x;
  std::memcpy(&x, &u, 8);
  return x;
#endif
}

__host__ __device__ __forceinline__ float bitsf(uint32_t u) {
#ifdef __CUDA_ARCH__
  return __uint_as_float(u);
#else
  float x;
  std::memcpy(&x, &u, 4);
  return x;
#endif
}

__host__ __device__ __forceinline__ uint32_t fbits(float x) {
#ifdef __CUDA_ARCH__
  return (uint32_t)__float_as_uint(x);
#else
  uint32_t u;
  std::memcpy(&u, &x, 4);
  return u;
#endif
}

// Correctly rounded 1/b for every b whose reciprocal is a normal number and
// whose significand is not a power of two: *special is set for zeros,
// subnormals, infinities, NaN and |b| >= 2^1021, and the value returned then is
// meaningless.  Straight-line code (no branches), so it interleaves with other
// work.
__host__ __device__ __forceinline__ double rcp_rn_fast(double b, bool *special) {
  const uint64_t bits = dbits(b);
  const uint64_t E = (bits >> 52) & 0x7ffull;
  const uint64_t frac = bits & ((1ull << 52) - 1);
  const uint64_t sign = bits & (1ull << 63);
  *special = (E == 0) | (E >= 2045);
  const uint64_t m = frac | (1ull << 52);
  // M = m / 2^29 = xh + xl/2^29 with xh = floor(M), 2^23 <= xh < 2^24, written straight
  // into a float's bits (exponent 2^23), and 0 <= xl < 2^29.
  const uint32_t xh = (uint32_t)(m >> 29);
  const int32_t xl = (int32_t)(m & ((1ull << 29) - 1));
  const float xhf = bitsf((150u << 23) | (xh & 0x7fffffu)), xlf = (float)xl * 0x1p-29f;
  // y ~ 1/xh: hardware seed plus one Newton step; then one Newton step for 1/M
  // carried as the unevaluated pair y + t (relative error below 2^-45, plus 2^-47 from
  // rounding xl to a float).
  const float y0 = rcp_approx_f32(xhf);
  const float y = fmaf(y0, fmaf(-xhf, y0, 1.0f), y0);
  const float e = fmaf(-xlf, y, fmaf(-xhf, y, 1.0f));  // 1 - M*y
  const float t = y * e;
  // Q = (y + t) * 2^76 ~ 2^105/m within 2^9; y*2^76 is an exact integer (y in [2^-24, 2^-23]).
  const uint32_t yb = fbits(y);
  const uint32_t ym = (yb & 0x7fffffu) | 0x800000u;  // y = ym * 2^(yexp - 150)
  const int yexp = (int)(yb >> 23);
  uint64_t Q = (uint64_t)ym << (yexp - 74);
  Q = (uint64_t)((int64_t)Q + (int64_t)(int32_t)(t * 0x1p76f));
  // one correction from the exact remainder (2^105 = 0 mod 2^64 and |R| < 2^62): Q += R/m,
  // R/m ~ (R >> 31) * y * 2^2 = (R >> 31) * ym / 2^(148 - yexp), floored, within one unit
  int64_t R = (int64_t)(0ull - Q * m);
  Q = (uint64_t)((int64_t)Q + (((int64_t)(int32_t)(R >> 31) * (int64_t)ym) >> (148 - yexp)));
  // now |Q - 2^105/m| < 1.01: the exact remainder fixes Q and decides the rounding
  R = (int64_t)(0ull - Q * m);
  const bool lo = R < 0, hi = R >= (int64_t)m;
  Q = lo ? Q - 1 : (hi ? Q + 1 : Q);
  R = lo ? R + (int64_t)m : (hi ? R - (int64_t)m : R);
  Q += ((uint64_t)R > m - (uint64_t)R) ? 1ull : 0ull;  // 2R > m: round up
  const uint64_t rbits = sign | ((2045 - E) << 52) | (Q - (1ull << 52));
  const uint64_t pbits = sign | ((2046 - E) << 52);  // significand 1: 1/b is a power of two
  return bitsd(frac == 0 ? pbits : rbits);
}

#ifdef __CUDACC__
// Out of line, so that the rarely taken division is never if-converted (an
// unconditional FP64 division in every thread costs more than the reciprocal).
__device__ __noinline__ static double rcp_division(double b) { return 1.0 / b; }
#endif

// Correctly rounded 1/b (IEEE binary64, round to nearest even).
__host__ __device__ __forceinline__ double rcp_rn(double b) {
  bool special;
  double r = rcp_rn_fast(b, &special);
#ifdef __CUDA_ARCH__
  if (special) r = rcp_division(b);
#else
  if (special) r = 1.0 / b;
#endif
  return r;
}

// ---------------------------------------------------------------------------
// x / d, correctly rounded, for a divisor known before the dividend (the
// diagonal of U in the back substitution).  Ahead of time, off the dependence
// chain, d gets a two-term reciprocal (div_known_prep):
//   yh = RN(1/d)                      (rcp_rn)
//   yl = RN(RN(1 - d*yh) * yh)        1 - d*yh is exact for a correctly rounded
//                                     yh, so yh + yl = 1/d within ~2^-104 relative.
// The quotient then takes four dependent floating-point operations instead of
// a full division (Markstein's final step: P. Markstein, IBM J. Res. Dev.
// 34(1), 1990):
//   q0 = RN(x*yh + RN(x*yl))          within half an ulp plus 2^-50 ulp of x/d:
//                                     a faithful quotient
//   q  = RN(q0 + (x - d*q0)*yh)       x - d*q0 is exact for a faithful q0, and with
//                                     yh correctly rounded this returns RN(x/d)
// (Markstein's theorem).  No quotient of two binary64 numbers lies on a
// rounding midpoint, so the result is the IEEE quotient bit for bit.  The
// theorem assumes that no step overflows or underflows: div_known keeps to
// biased exponents 64..1983 for x and d with |E(x) - E(d)| <= 900 (quotient
// exponent within 2^-900..2^901, every remainder far above the subnormal range)
// and takes the ordinary division otherwise (zeros, subnormals, infinities,
// NaN, huge or tiny ratios).
__host__ __device__ __forceinline__ int dexp(double x) { return (int)((dbits(x) >> 52) & 0x7ffull); }

// Two-term reciprocal of d; *ok tells whether d is inside the range div_known
// handles (when it is not, yh and yl are not used).
__host__ __device__ __forceinline__ void div_known_prep(double d, double *yh, double *yl, bool *ok) {
  const int e = dexp(d);
  *ok = e >= 64 && e <= 1983;
  const double h = rcp_rn(d);
  *yh = h;
  *yl = *ok ? fma(-d, h, 1.0) * h : 0.0;
}

#ifdef __CUDACC__
__device__ __noinline__ static double div_division(double x, double d) { return x / d; }
#endif

// x / d given div_known_prep(d, &yh, &yl, &d_ok).
__host__ __device__ __forceinline__ double div_known(double x, double d, double yh, double yl, bool d_ok) {
  const int ex = dexp(x), ed = dexp(d);
  const bool ok = d_ok && ex >= 64 && ex <= 1983 && ex - ed <= 900 && ed - ex <= 900;
  const double t = x * yl;
  double q = fma(x, yh, t);
  const double r = fma(-q, d, x);
  q = fma(r, yh, q);
  if (!ok) {
#ifdef __CUDA_ARCH__
    q = div_division(x, d);
#else
    q = x / d;
#endif
  }
  return q;
}

// The back substitution's quotient with the reference-BLAS zero test: x / d for a
// nonzero x (div_known), x itself for a zero x (no division, its sign kept).  The
// four-operation path is computed without a branch on x; a zero x fails its
// exponent-range test and takes the (rare) fallback.
__host__ __device__ __forceinline__ double div_known_nz(double x, double d, double yh, double yl, bool d_ok) {
  const int ex = dexp(x), ed = dexp(d);
  const bool ok = d_ok && ex >= 64 && ex <= 1983 && ex - ed <= 900 && ed - ex <= 900;
  const double t = x * yl;
  double q = fma(x, yh, t);
  const double r = fma(-q, d, x);
  q = fma(r, yh, q);
  if (!ok) {
    if (x != 0.0) {
#ifdef __CUDA_ARCH__
      q = div_division(x, d);
#else
      q = x / d;
#endif
    } else {
      q = x;
    }
  }
  return q;
}

}  // namespace bandlu
