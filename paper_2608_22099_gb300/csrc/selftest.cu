// selftest.cu -- self-test hooks (declared in include/bandlu_selftest.h): the
// integer-pipe reciprocal used on the pivot chain and the known-divisor division
// of the back substitution, callable on the host and on the device so tests can
// compare them bit for bit with IEEE division (and the quotient with its zero test
// on the host).
#include "bandlu_selftest.h"
#include "common.cuh"
#include "rcp.cuh"

namespace {
__global__ void k_rcp(const double *__restrict__ x, double *__restrict__ y, long long n) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
    y[i] = bandlu::rcp_rn(x[i]);
}
__global__ void k_div(const double *__restrict__ x, double *__restrict__ y, long long n) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
    y[i] = 1.0 / x[i];
}
__global__ void k_divk(const double *__restrict__ x, const double *__restrict__ d, double *__restrict__ q,
                       long long n, int use_division) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    if (use_division) {
      q[i] = x[i] / d[i];
    } else {
      double yh, yl;
      bool ok;
      bandlu::div_known_prep(d[i], &yh, &yl, &ok);
      q[i] = bandlu::div_known(x[i], d[i], yh, yl, ok);
    }
  }
}
}  // namespace

extern "C" {

void bandlu_selftest_div_host(const double *x, const double *d, double *q, int64_t n) {
  for (int64_t i = 0; i < n; ++i) {
    double yh, yl;
    bool ok;
    bandlu::div_known_prep(d[i], &yh, &yl, &ok);
    q[i] = bandlu::div_known(x[i], d[i], yh, yl, ok);
  }
}

void bandlu_selftest_div_nz_host(const double *x, const double *d, double *q, int64_t n) {
  for (int64_t i = 0; i < n; ++i) {
    double yh, yl;
    bool ok;
    bandlu::div_known_prep(d[i], &yh, &yl, &ok);
    q[i] = bandlu::div_known_nz(x[i], d[i], yh, yl, ok);
  }
}

int bandlu_selftest_div_device(const double *x, const double *d, double *q, int64_t n, int use_division,
                               cudaStream_t stream) {
  if (n < 0) return -4;
  if (n == 0) return BANDLU_OK;
  if (x == nullptr) return -1;
  if (d == nullptr) return -2;
  if (q == nullptr) return -3;
  long long blocks = (n + 255) / 256;
  if (blocks > 152ll * 64) blocks = 152ll * 64;
  k_divk<<<(unsigned)blocks, 256, 0, stream>>>(x, d, q, n, use_division);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

void bandlu_selftest_rcp_host(const double *x, double *y, int64_t n) {
  for (int64_t i = 0; i < n; ++i) y[i] = bandlu::rcp_rn(x[i]);
}

int bandlu_selftest_rcp_device(const double *x, double *y, int64_t n, int use_division, cudaStream_t stream) {
  if (n < 0) return -3;
  if (n == 0) return BANDLU_OK;
  if (x == nullptr) return -1;
  if (y == nullptr) return -2;
  long long blocks = (n + 255) / 256;
  if (blocks > 152ll * 64) blocks = 152ll * 64;
  if (use_division)
    k_div<<<(unsigned)blocks, 256, 0, stream>>>(x, y, n);
  else
    k_rcp<<<(unsigned)blocks, 256, 0, stream>>>(x, y, n);
  BANDLU_CHECK_LAUNCH();
  return BANDLU_OK;
}

}  // extern "C"
