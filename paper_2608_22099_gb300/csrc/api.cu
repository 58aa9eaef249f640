// api.cu -- the C ABI (declared in include/bandlu.h): argument checks, then the
// launches of detect.cu, convert.cu, gbtrf.cu, gbtrf_wide.cu, gbtrs.cu,
// trsolve.cu and batched.cu.
#include <climits>
#include <mutex>
#include <set>
#include <utility>

#include "common.cuh"

namespace bandlu {

bool allow_dynamic_smem(const void *kernel, int bytes) {
  static std::mutex mu;
  static std::set<std::pair<const void *, int>> done;  // (kernel, device) pairs already opted in
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  std::lock_guard<std::mutex> lock(mu);
  if (done.count({kernel, dev})) return true;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess) return false;
  done.insert({kernel, dev});
  return true;
}

int device_sms() {
  constexpr int kMaxDev = 64;
  static std::mutex mu;
  static int sms[kMaxDev] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 152;
  if (dev < 0 || dev >= kMaxDev) {
    int v = 0;
    return cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0 ? v : 152;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (sms[dev] == 0) {
    int v = 0;
    sms[dev] = cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0 ? v : 152;
  }
  return sms[dev];
}

}  // namespace bandlu

namespace {

inline bool bad_n(int64_t n) { return n < 0 || n > (int64_t)INT_MAX; }
inline int64_t max1(int64_t n) { return n > 1 ? n : 1; }
// a leading dimension whose n columns' (or rows') extent n * ld would not fit
// the 64-bit offsets the kernels compute
inline bool bad_ld(int64_t n, int64_t ld) { return ld < max1(n) || ld > INT64_MAX / max1(n); }
// an extent ld per item that would overflow 64-bit offsets over count items
inline bool too_long(int64_t count, int64_t ld) { return ld > INT64_MAX / max1(count); }
// the same for strides between the matrices of a batch
inline bool bad_stride(int64_t count, int64_t stride, int64_t minimum) {
  return stride < minimum || (count > 0 && stride > INT64_MAX / count);
}

}  // namespace

extern "C" {

const char *bandlu_version(void) { return "bandlu 0.1 (sm_103a)"; }

int detect_bandwidth(const double *A, int64_t n, int64_t lda, int *d_kl, int *d_ku, cudaStream_t stream) {
  if (bad_n(n)) return -2;
  if (A == nullptr && n > 0) return -1;
  if (bad_ld(n, lda)) return -3;
  if (d_kl == nullptr) return -4;
  if (d_ku == nullptr) return -5;
  return bandlu::launch_detect(A, n, lda, d_kl, d_ku, stream);
}

int dense_to_band(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                  cudaStream_t stream) {
  if (bad_n(n)) return -3;
  if (A == nullptr && n > 0) return -1;
  if (bad_ld(n, lda)) return -2;
  if (kl < 0) return -4;
  if (ku < 0) return -5;
  if (AB == nullptr && n > 0) return -6;
  if (ldab < 2 * (int64_t)kl + ku + 1 || too_long(n, ldab)) return -7;
  return bandlu::launch_dense_to_band(A, lda, n, kl, ku, AB, ldab, stream);
}

int detect_bandwidth_cm(const double *A, int64_t n, int64_t lda, int *d_kl, int *d_ku, cudaStream_t stream) {
  if (bad_n(n)) return -2;
  if (A == nullptr && n > 0) return -1;
  if (bad_ld(n, lda)) return -3;
  if (d_kl == nullptr) return -4;
  if (d_ku == nullptr) return -5;
  // read as row-major, the column-major A is its transpose: the lower and upper
  // bandwidths trade places
  return bandlu::launch_detect(A, n, lda, d_ku, d_kl, stream);
}

int dense_to_band_cm(const double *A, int64_t lda, int64_t n, int kl, int ku, double *AB, int64_t ldab,
                     cudaStream_t stream) {
  if (bad_n(n)) return -3;
  if (A == nullptr && n > 0) return -1;
  if (bad_ld(n, lda)) return -2;
  if (kl < 0) return -4;
  if (ku < 0) return -5;
  if (AB == nullptr && n > 0) return -6;
  if (ldab < 2 * (int64_t)kl + ku + 1 || too_long(n, ldab)) return -7;
  return bandlu::launch_dense_to_band_cm(A, lda, n, kl, ku, AB, ldab, stream);
}

int gbtrf(int64_t n, int kl, int ku, double *AB, int64_t ldab, int *ipiv, int *d_info, cudaStream_t stream) {
  if (bad_n(n)) return -1;
  if (kl < 0) return -2;
  if (ku < 0) return -3;
  if (AB == nullptr && n > 0) return -4;
  if (ldab < 2 * (int64_t)kl + ku + 1 || too_long(n, ldab)) return -5;
  if (ipiv == nullptr && n > 0) return -6;
  if (d_info == nullptr) return -7;
  return bandlu::launch_gbtrf(n, kl, ku, AB, ldab, ipiv, d_info, stream);
}

int dispatch_lu(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *h_kl, int *h_ku,
                int *d_info, cudaStream_t stream) {
  if (A == nullptr && n > 0) return -1;
  if (bad_n(n)) return -2;
  if (bad_ld(n, lda)) return -3;
  if (AB == nullptr && n > 0) return -4;
  if (ldab < 1 || too_long(n, ldab)) return -5;
  if (ipiv == nullptr && n > 0) return -6;
  if (h_kl == nullptr) return -7;
  if (h_ku == nullptr) return -8;
  if (d_info == nullptr) return -9;
  int *d_klku = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&d_klku), 2 * sizeof(int), stream) != cudaSuccess)
    return BANDLU_ERR_CUDA;
  int rc = bandlu::launch_detect(A, n, lda, d_klku, d_klku + 1, stream);
  int h[2] = {0, 0};
  if (rc == BANDLU_OK && cudaMemcpyAsync(h, d_klku, sizeof(h), cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    rc = BANDLU_ERR_CUDA;
  if (cudaFreeAsync(d_klku, stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (rc != BANDLU_OK) return rc;
  *h_kl = h[0];
  *h_ku = h[1];
  if (!bandlu::predicate_banded(n, h[0], h[1], ldab)) return BANDLU_NOT_BANDED;
  rc = bandlu::launch_dense_to_band(A, lda, n, h[0], h[1], AB, ldab, stream);
  if (rc != BANDLU_OK) return rc;
  return bandlu::launch_gbtrf(n, h[0], h[1], AB, ldab, ipiv, d_info, stream);
}

int dispatch_lu_cm(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *h_kl,
                   int *h_ku, int *d_info, cudaStream_t stream) {
  if (A == nullptr && n > 0) return -1;
  if (bad_n(n)) return -2;
  if (bad_ld(n, lda)) return -3;
  if (AB == nullptr && n > 0) return -4;
  if (ldab < 1 || too_long(n, ldab)) return -5;
  if (ipiv == nullptr && n > 0) return -6;
  if (h_kl == nullptr) return -7;
  if (h_ku == nullptr) return -8;
  if (d_info == nullptr) return -9;
  int *d_klku = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&d_klku), 2 * sizeof(int), stream) != cudaSuccess)
    return BANDLU_ERR_CUDA;
  int rc = bandlu::launch_detect(A, n, lda, d_klku + 1, d_klku, stream);  // transposed view: (ku, kl)
  int h[2] = {0, 0};
  if (rc == BANDLU_OK && cudaMemcpyAsync(h, d_klku, sizeof(h), cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    rc = BANDLU_ERR_CUDA;
  if (cudaFreeAsync(d_klku, stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (rc != BANDLU_OK) return rc;
  *h_kl = h[0];
  *h_ku = h[1];
  if (!bandlu::predicate_banded(n, h[0], h[1], ldab)) return BANDLU_NOT_BANDED;
  rc = bandlu::launch_dense_to_band_cm(A, lda, n, h[0], h[1], AB, ldab, stream);
  if (rc != BANDLU_OK) return rc;
  return bandlu::launch_gbtrf(n, h[0], h[1], AB, ldab, ipiv, d_info, stream);
}

int dispatch_lu_async(const double *A, int64_t n, int64_t lda, double *AB, int64_t ldab, int *ipiv, int *d_kl,
                      int *d_ku, int *d_status, int *d_info, cudaStream_t stream) {
  if (A == nullptr && n > 0) return -1;
  if (bad_n(n)) return -2;
  if (bad_ld(n, lda)) return -3;
  if (AB == nullptr && n > 0) return -4;
  if (ldab < 1 || ldab > (int64_t)INT_MAX) return -5;
  if (ipiv == nullptr && n > 0) return -6;
  if (d_kl == nullptr) return -7;
  if (d_ku == nullptr) return -8;
  if (d_status == nullptr) return -9;
  if (d_info == nullptr) return -10;
  int rc = bandlu::launch_detect(A, n, lda, d_kl, d_ku, stream);
  if (rc == BANDLU_OK) rc = bandlu::launch_decide_convert(A, lda, n, ldab, d_kl, d_ku, d_status, AB, stream);
  if (rc == BANDLU_OK) rc = bandlu::launch_gbtrf_on_device(n, AB, ldab, ipiv, d_kl, d_ku, d_status, d_info, stream);
  return rc;
}

int gbtrs(int64_t n, int kl, int ku, int64_t nrhs, const double *AB, int64_t ldab, const int *ipiv, double *B,
          int64_t ldb, cudaStream_t stream) {
  const bool work = n > 0 && nrhs > 0;
  if (bad_n(n)) return -1;
  if (kl < 0) return -2;
  if (ku < 0) return -3;
  if (nrhs < 0 || nrhs > (int64_t)INT_MAX) return -4;
  if (AB == nullptr && work) return -5;
  if (ldab < 2 * (int64_t)kl + ku + 1 || too_long(n, ldab)) return -6;
  if (ipiv == nullptr && work) return -7;
  if (B == nullptr && work) return -8;
  if (ldb < max1(n) || too_long(nrhs, ldb)) return -9;
  return bandlu::launch_gbtrs(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, nullptr, stream);
}

int dispatch_solve(const double *A, int64_t n, int64_t lda, double *B, int64_t ldb, int64_t nrhs, double *AB,
                   int64_t ldab, int *ipiv, int *h_kl, int *h_ku, int *d_info, cudaStream_t stream) {
  const bool work = n > 0 && nrhs > 0;
  if (A == nullptr && n > 0) return -1;
  if (bad_n(n)) return -2;
  if (bad_ld(n, lda)) return -3;
  if (B == nullptr && work) return -4;
  if (ldb < max1(n) || too_long(nrhs, ldb)) return -5;
  if (nrhs < 0 || nrhs > (int64_t)INT_MAX) return -6;
  if (AB == nullptr && n > 0) return -7;
  if (ldab < 1 || too_long(n, ldab)) return -8;
  if (ipiv == nullptr && n > 0) return -9;
  if (h_kl == nullptr) return -10;
  if (h_ku == nullptr) return -11;
  if (d_info == nullptr) return -12;
  const int rc = dispatch_lu(A, n, lda, AB, ldab, ipiv, h_kl, h_ku, d_info, stream);
  if (rc != BANDLU_OK) return rc;  // BANDLU_NOT_BANDED: B untouched, the caller solves densely
  // the solve reads info on the device and leaves B as it is for a singular factor
  return bandlu::launch_gbtrs(n, *h_kl, *h_ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, stream);
}

int trsv_band(int lower, int64_t n, int k, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs,
              int *d_info, cudaStream_t stream) {
  const bool work = n > 0 && nrhs > 0;
  if (lower != 0 && lower != 1) return -1;
  if (bad_n(n)) return -2;
  if (k < 0 || (n > 0 && k > n - 1)) return -3;
  if (A == nullptr && n > 0) return -4;
  if (bad_ld(n, lda)) return -5;
  if (B == nullptr && work) return -6;
  if (ldb < max1(n) || too_long(nrhs, ldb)) return -7;
  if (nrhs < 0 || nrhs > (int64_t)INT_MAX) return -8;
  if (d_info == nullptr) return -9;
  return bandlu::launch_trsv(lower == 1, n, k, A, lda, B, ldb, nrhs, d_info, stream);
}

int diag_solve(int64_t n, const double *A, int64_t lda, double *B, int64_t ldb, int64_t nrhs, int *d_info,
               cudaStream_t stream) {
  const bool work = n > 0 && nrhs > 0;
  if (bad_n(n)) return -1;
  if (A == nullptr && n > 0) return -2;
  if (bad_ld(n, lda)) return -3;
  if (B == nullptr && work) return -4;
  if (ldb < max1(n) || too_long(nrhs, ldb)) return -5;
  if (nrhs < 0 || nrhs > (int64_t)INT_MAX) return -6;
  if (d_info == nullptr) return -7;
  return bandlu::launch_diag_solve(n, A, lda, B, ldb, nrhs, d_info, stream);
}

int bandlu_classify(int64_t n, int kl, int ku, int64_t ldab) {
  if (n < 0 || kl < 0 || ku < 0) return -1;
  if (ku == 0) return kl == 0 ? BANDLU_KIND_DIAGONAL : BANDLU_KIND_LOWER;
  if (kl == 0) return BANDLU_KIND_UPPER;
  return bandlu::predicate_banded(n, kl, ku, ldab) ? BANDLU_KIND_BANDED : BANDLU_KIND_DENSE;
}

int dispatch_backslash(const double *A, int64_t n, int64_t lda, double *B, int64_t ldb, int64_t nrhs, double *AB,
                       int64_t ldab, int *ipiv, int *h_kl, int *h_ku, int *h_kind, int *d_info, cudaStream_t stream) {
  const bool work = n > 0 && nrhs > 0;
  if (A == nullptr && n > 0) return -1;
  if (bad_n(n)) return -2;
  if (bad_ld(n, lda)) return -3;
  if (B == nullptr && work) return -4;
  if (ldb < max1(n) || too_long(nrhs, ldb)) return -5;
  if (nrhs < 0 || nrhs > (int64_t)INT_MAX) return -6;
  if (AB == nullptr && n > 0) return -7;
  if (ldab < 1 || too_long(n, ldab)) return -8;
  if (ipiv == nullptr && n > 0) return -9;
  if (h_kl == nullptr) return -10;
  if (h_ku == nullptr) return -11;
  if (h_kind == nullptr) return -12;
  if (d_info == nullptr) return -13;
  int *d_klku = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&d_klku), 2 * sizeof(int), stream) != cudaSuccess)
    return BANDLU_ERR_CUDA;
  int rc = bandlu::launch_detect(A, n, lda, d_klku, d_klku + 1, stream);
  int h[2] = {0, 0};
  if (rc == BANDLU_OK && cudaMemcpyAsync(h, d_klku, sizeof(h), cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    rc = BANDLU_ERR_CUDA;
  if (cudaFreeAsync(d_klku, stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess && rc == BANDLU_OK) rc = BANDLU_ERR_CUDA;
  if (rc != BANDLU_OK) return rc;
  const int kl = h[0], ku = h[1];
  *h_kl = kl;
  *h_ku = ku;
  const int kind = bandlu_classify(n, kl, ku, ldab);
  *h_kind = kind;
  switch (kind) {
    case BANDLU_KIND_DIAGONAL:
      return bandlu::launch_diag_solve(n, A, lda, B, ldb, nrhs, d_info, stream);
    case BANDLU_KIND_LOWER:
      return bandlu::launch_trsv(true, n, kl, A, lda, B, ldb, nrhs, d_info, stream);
    case BANDLU_KIND_UPPER:
      return bandlu::launch_trsv(false, n, ku, A, lda, B, ldb, nrhs, d_info, stream);
    case BANDLU_KIND_BANDED:
      rc = bandlu::launch_dense_to_band(A, lda, n, kl, ku, AB, ldab, stream);
      if (rc == BANDLU_OK) rc = bandlu::launch_gbtrf(n, kl, ku, AB, ldab, ipiv, d_info, stream);
      if (rc == BANDLU_OK) rc = bandlu::launch_gbtrs(n, kl, ku, nrhs, AB, ldab, ipiv, B, ldb, d_info, stream);
      return rc;
    default:
      return BANDLU_NOT_BANDED;  // B untouched: the caller's dense LU
  }
}

int dispatch_lu_batched(const double *A, int64_t n, int64_t lda, int64_t strideA, int64_t batch, double *AB,
                        int64_t ldab, int64_t strideAB, int *ipiv, int64_t strideP, int *d_kl, int *d_ku,
                        int *d_info, int *d_status, cudaStream_t stream) {
  const bool work = n > 0 && batch > 0;
  if (A == nullptr && work) return -1;
  if (bad_n(n)) return -2;
  if (bad_ld(n, lda)) return -3;
  if (bad_stride(batch, strideA, n * lda)) return -4;
  if (batch < 0) return -5;
  if (AB == nullptr && work) return -6;
  if (ldab < 1 || ldab > (int64_t)INT_MAX) return -7;
  if (bad_stride(batch, strideAB, n * ldab)) return -8;
  if (ipiv == nullptr && work) return -9;
  if (bad_stride(batch, strideP, n)) return -10;
  if ((d_kl == nullptr || d_ku == nullptr || d_info == nullptr || d_status == nullptr) && batch > 0) {
    if (d_kl == nullptr) return -11;
    if (d_ku == nullptr) return -12;
    if (d_info == nullptr) return -13;
    return -14;
  }
  return bandlu::launch_batched(A, n, lda, strideA, batch, AB, ldab, strideAB, ipiv, strideP, d_kl, d_ku, d_info,
                                d_status, stream);
}

}  // extern "C"
