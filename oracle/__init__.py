"""CPU oracle for the structure-aware banded LU dispatch (Lujan & Edelman, HPEC 2025).

TEST INFRASTRUCTURE ONLY.  The functions here are the independent reference the
CUDA path is checked against.  Only the test suite, ``__graft_entry__.smoke()``
and the benchmark's CPU-baseline leg may import this package; the CUDA library
and its Python binding never do.

The arithmetic lives in ``bandlu_oracle.c`` (plain C, IEEE binary64, built with
``-ffp-contract=off``); this module compiles it with gcc on first use and wraps
it with ctypes over numpy arrays.

Layouts: ``A`` is a dense row-major ``(n, lda)`` float64 array (only the first
``n`` columns are the matrix); ``AB`` is LAPACK band storage, column-major
``ldab x n``, held here as a numpy array of shape ``(n, ldab)`` whose row ``j``
is band column ``j`` (so ``AB[j, r]`` is ``AB(r, j)``); ``ipiv`` is 1-based.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bandlu_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle_bandlu.so")
# Timing build only: the same source compiled with OpenMP, whose pragmas split the
# detection scan and the conversion over rows/columns and a batch over its
# matrices.  Nothing in the arithmetic changes (a max-reduction, plain copies and
# independent matrices); the pinned, checked library is the single-threaded one.
_OMP_LIB_PATH = os.path.join(_BUILD, "liboracle_bandlu_omp.so")
_lock = threading.Lock()
_lib = None
_omp_lib = None

CFLAGS = ["-O2", "-fPIC", "-shared", "-std=gnu11", "-ffp-contract=off", "-fno-fast-math"]


def build(force: bool = False, omp: bool = False) -> str:
    """Compile the oracle with gcc into ``oracle/_build``; returns the .so path.
    omp=True builds the OpenMP timing variant (used only to time the CPU baseline)."""
    os.makedirs(_BUILD, exist_ok=True)
    path = _OMP_LIB_PATH if omp else _LIB_PATH
    if (not force and os.path.exists(path)
            and os.path.getmtime(path) >= os.path.getmtime(_SRC)):
        return path
    tmp = path + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *CFLAGS, *(["-fopenmp"] if omp else []), "-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, path)
    return path


def _load(omp: bool = False):
    global _lib, _omp_lib
    with _lock:
        if omp and _omp_lib is not None:
            return _omp_lib
        if not omp and _lib is not None:
            return _lib
        if omp:
            path = build(omp=True)
        else:
            # A mutation test points this at a deliberately broken build of the oracle to show
            # that the pins catch the mistake; normal use leaves it unset.
            path = os.environ.get("BANDLU_ORACLE_LIB") or build()
        lib = ctypes.CDLL(path)
        i64, i32, dp, ip = ctypes.c_int64, ctypes.c_int, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int)
        i64p = ctypes.POINTER(ctypes.c_int64)
        lib.oracle_detect_bandwidth.argtypes = [dp, i64, i64, ip, ip]
        lib.oracle_dense_to_band.argtypes = [dp, i64, i64, i32, i32, dp, i64]
        lib.oracle_band_to_dense.argtypes = [i64, i32, i32, dp, i64, dp, i64]
        lib.oracle_gbtrf.argtypes = [i64, i32, i32, dp, i64, ip, i64p]
        lib.oracle_getrf_dense.argtypes = [i64, dp, i64, ip]
        lib.oracle_band_residual.argtypes = [i64, i32, i32, dp, i64, dp, i64, ip, dp, dp]
        lib.oracle_band_residual.restype = ctypes.c_double
        lib.oracle_is_banded.argtypes = [i64, i32, i32, i64]
        lib.oracle_gbtrs.argtypes = [i64, i32, i32, i64, dp, i64, ip, dp, i64]
        lib.oracle_dispatch_lu_batched.argtypes = [dp, i64, i64, i64, i64, dp, i64, i64, ip, i64, ip, ip, ip, ip]
        lib.oracle_dispatch_lu_batched.restype = None
        lib.oracle_detect_bandwidth_cm.argtypes = [dp, i64, i64, ip, ip]
        lib.oracle_dense_to_band_cm.argtypes = [dp, i64, i64, i32, i32, dp, i64]
        lib.oracle_tbsv_dense.argtypes = [i32, i64, i64, dp, i64, i64, dp, i64, ip]
        lib.oracle_diag_solve.argtypes = [i64, dp, i64, i64, dp, i64, ip]
        lib.oracle_classify.argtypes = [i64, i32, i32, i64]
        lib.oracle_dispatch_backslash.argtypes = [dp, i64, i64, dp, i64, i64, dp, i64, ip, ip, ip, ip, ip]
        if omp:
            _omp_lib = lib
        else:
            _lib = lib
        return lib


def _dptr(a: np.ndarray):
    assert a.dtype == np.float64 and a.flags.c_contiguous
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _iptr(a: np.ndarray):
    assert a.dtype == np.int32 and a.flags.c_contiguous
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


def _dense(A: np.ndarray):
    A = np.ascontiguousarray(A, dtype=np.float64)
    n, lda = A.shape[0], A.shape[1]
    assert lda >= n
    return A, n, lda


def ldab_for(kl: int, ku: int) -> int:
    """Height of LAPACK band storage with room for pivoting fill: 2*kl+ku+1."""
    return 2 * kl + ku + 1


def detect_bandwidth(A: np.ndarray, omp: bool = False) -> tuple[int, int]:
    """(kl, ku) of the n x n row-major matrix held in ``A[:, :n]`` (omp: the timing build)."""
    A, n, lda = _dense(A)
    kl, ku = ctypes.c_int(), ctypes.c_int()
    rc = _load(omp).oracle_detect_bandwidth(_dptr(A), n, max(lda, 1), ctypes.byref(kl), ctypes.byref(ku))
    if rc != 0:
        raise ValueError("oracle_detect_bandwidth: bad argument")
    return kl.value, ku.value


def dense_to_band(A: np.ndarray, kl: int, ku: int, ldab: int | None = None, omp: bool = False) -> np.ndarray:
    """Band storage of A as an (n, ldab) array: ``AB[j, kl+ku+i-j] = A[i, j]`` (omp: the timing build)."""
    A, n, lda = _dense(A)
    ldab = ldab_for(kl, ku) if ldab is None else ldab
    AB = np.empty((n, ldab), dtype=np.float64)
    rc = _load(omp).oracle_dense_to_band(_dptr(A), n, max(lda, 1), kl, ku, _dptr(AB), ldab)
    if rc != 0:
        raise ValueError("oracle_dense_to_band: bad argument")
    return AB


def band_to_dense(AB: np.ndarray, kl: int, ku: int) -> np.ndarray:
    AB = np.ascontiguousarray(AB, dtype=np.float64)
    n, ldab = AB.shape
    A = np.empty((n, n), dtype=np.float64)
    rc = _load().oracle_band_to_dense(n, kl, ku, _dptr(AB), ldab, _dptr(A), max(n, 1))
    if rc != 0:
        raise ValueError("oracle_band_to_dense: bad argument")
    return A


def gbtrf(AB: np.ndarray, kl: int, ku: int) -> tuple[np.ndarray, np.ndarray, int, int]:
    """Factor a copy of the band; returns (AB_factored, ipiv (1-based int32), info, flops)."""
    AB = np.array(AB, dtype=np.float64, order="C", copy=True)
    n, ldab = AB.shape
    ipiv = np.zeros(n, dtype=np.int32)
    fl = ctypes.c_int64()
    info = _load().oracle_gbtrf(n, kl, ku, _dptr(AB), ldab, _iptr(ipiv), ctypes.byref(fl))
    if info < 0:
        raise ValueError("oracle_gbtrf: bad argument")
    return AB, ipiv, info, fl.value


def gbtrs(ABf: np.ndarray, ipiv: np.ndarray, kl: int, ku: int, B: np.ndarray) -> np.ndarray:
    """Solve A X = B with the factors of gbtrf; B (and the result) has shape (nrhs, ldb), row c
    being right-hand side c (column-major ldb x nrhs storage).  Returns X."""
    ABf = np.ascontiguousarray(ABf, dtype=np.float64)
    ipiv = np.ascontiguousarray(ipiv, dtype=np.int32)
    X = np.array(B, dtype=np.float64, order="C", copy=True)
    if X.ndim == 1:
        X = X[None]
    n, ldab = ABf.shape
    nrhs, ldb = X.shape
    rc = _load().oracle_gbtrs(n, kl, ku, nrhs, _dptr(ABf), ldab, _iptr(ipiv), _dptr(X), max(ldb, 1))
    if rc != 0:
        raise ValueError("oracle_gbtrs: bad argument")
    return X


def getrf_dense(A: np.ndarray) -> tuple[np.ndarray, np.ndarray, int]:
    """Dense LU of a copy of A (row-major), interchanges over columns j..n-1 only."""
    A = np.array(A, dtype=np.float64, order="C", copy=True)
    n, lda = A.shape
    ipiv = np.zeros(n, dtype=np.int32)
    info = _load().oracle_getrf_dense(n, _dptr(A), max(lda, 1), _iptr(ipiv))
    if info < 0:
        raise ValueError("oracle_getrf_dense: bad argument")
    return A, ipiv, info


def band_residual(A: np.ndarray, ABf: np.ndarray, ipiv: np.ndarray, kl: int, ku: int) -> tuple[float, float]:
    """(||A - P0 L0 ... U||_inf, ||A||_inf) computed in band form."""
    A, n, lda = _dense(A)
    ABf = np.ascontiguousarray(ABf, dtype=np.float64)
    ipiv = np.ascontiguousarray(ipiv, dtype=np.int32)
    assert ABf.shape[0] == n
    W = np.empty(max(n * (2 * kl + ku + 1), 1), dtype=np.float64)
    an = ctypes.c_double()
    r = _load().oracle_band_residual(n, kl, ku, _dptr(A), max(lda, 1), _dptr(ABf), ABf.shape[1],
                                     _iptr(ipiv), _dptr(W), ctypes.byref(an))
    return r, an.value


def backward_error(A: np.ndarray, ABf: np.ndarray, ipiv: np.ndarray, kl: int, ku: int,
                   eps: float = 2.0 ** -53) -> float:
    """||A - P L U||_inf / (n * eps * ||A||_inf); eps defaults to the unit roundoff."""
    n = A.shape[0]
    r, an = band_residual(A, ABf, ipiv, kl, ku)
    if n == 0 or an == 0.0:
        return 0.0 if r == 0.0 else float("inf")
    return r / (n * eps * an)


def is_banded(n: int, kl: int, ku: int, ldab: int) -> bool:
    """The dispatch predicate: the speedup constraint (Eq. su-con) and the storage capacity."""
    return bool(_load().oracle_is_banded(n, kl, ku, ldab))


def dispatch_lu_batched(A: np.ndarray, ldab: int, omp: bool = False):
    """Batched dispatch over A of shape (batch, n, lda) (omp: the timing build, one matrix per thread).

    Returns dict with AB (batch, n, ldab), ipiv (batch, n), kl, ku, info, status
    (0 = factored, 1 = declined by the predicate).
    """
    A = np.ascontiguousarray(A, dtype=np.float64)
    batch, n, lda = A.shape
    AB = np.zeros((batch, n, ldab), dtype=np.float64)
    ipiv = np.zeros((batch, n), dtype=np.int32)
    kl = np.zeros(batch, dtype=np.int32)
    ku = np.zeros(batch, dtype=np.int32)
    info = np.zeros(batch, dtype=np.int32)
    status = np.zeros(batch, dtype=np.int32)
    _load(omp).oracle_dispatch_lu_batched(_dptr(A), n, max(lda, 1), n * lda, batch, _dptr(AB), ldab, n * ldab,
                                       _iptr(ipiv), n, _iptr(kl), _iptr(ku), _iptr(info), _iptr(status))
    return dict(AB=AB, ipiv=ipiv, kl=kl, ku=ku, info=info, status=status)


def dispatch_lu(A: np.ndarray, ldab: int):
    """Single-matrix dispatch (the batched routine with batch 1)."""
    A = np.ascontiguousarray(A, dtype=np.float64)
    r = dispatch_lu_batched(A[None], ldab)
    return dict(AB=r["AB"][0], ipiv=r["ipiv"][0], kl=int(r["kl"][0]), ku=int(r["ku"][0]),
                info=int(r["info"][0]), status=int(r["status"][0]))


# Kinds of the backslash dispatch (Listing 1), in the order it tests them.
KIND_DIAGONAL, KIND_LOWER, KIND_UPPER, KIND_BANDED, KIND_DENSE = 1, 2, 3, 4, 5


def _rhs(B: np.ndarray, n: int) -> np.ndarray:
    X = np.array(B, dtype=np.float64, order="C", copy=True)
    if X.ndim == 1:
        X = X[None]
    assert X.shape[1] >= n
    return X


def tbsv_dense(A: np.ndarray, lower: bool, k: int, B: np.ndarray) -> tuple[np.ndarray, int]:
    """Triangular solve with the band of width k of the (lower or upper) triangle of the
    row-major A; B (and the result) has shape (nrhs, ldb) as in gbtrs.  Returns (X, info);
    for info > 0 (a zero diagonal entry) X is B unchanged."""
    A, n, lda = _dense(A)
    X = _rhs(B, n)
    info = ctypes.c_int()
    rc = _load().oracle_tbsv_dense(1 if lower else 0, n, k, _dptr(A), max(lda, 1), X.shape[0], _dptr(X),
                                   max(X.shape[1], 1), ctypes.byref(info))
    if rc != 0:
        raise ValueError("oracle_tbsv_dense: bad argument")
    return X, info.value


def diag_solve(A: np.ndarray, B: np.ndarray) -> tuple[np.ndarray, int]:
    """X = B / diag(A) per right-hand side (rows of B); (X, info) as tbsv_dense."""
    A, n, lda = _dense(A)
    X = _rhs(B, n)
    info = ctypes.c_int()
    rc = _load().oracle_diag_solve(n, _dptr(A), max(lda, 1), X.shape[0], _dptr(X), max(X.shape[1], 1),
                                   ctypes.byref(info))
    if rc != 0:
        raise ValueError("oracle_diag_solve: bad argument")
    return X, info.value


def classify(n: int, kl: int, ku: int, ldab: int) -> int:
    """The branch of Listing 1 for bandwidths (kl, ku): one of the KIND_* values."""
    return int(_load().oracle_classify(n, kl, ku, ldab))


def dispatch_backslash(A: np.ndarray, B: np.ndarray, ldab: int):
    """A X = B through the backslash dispatch.  Returns dict with X (nrhs, n), kind, kl, ku,
    info, and AB, ipiv (the factors, meaningful for KIND_BANDED)."""
    A, n, lda = _dense(A)
    X = _rhs(B, n)
    AB = np.zeros((max(n, 1), ldab), dtype=np.float64)
    ipiv = np.zeros(max(n, 1), dtype=np.int32)
    kl, ku, kind, info = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    rc = _load().oracle_dispatch_backslash(_dptr(A), n, max(lda, 1), _dptr(X), max(X.shape[1], 1), X.shape[0],
                                           _dptr(AB), ldab, _iptr(ipiv), ctypes.byref(kl), ctypes.byref(ku),
                                           ctypes.byref(kind), ctypes.byref(info))
    if rc != 0:
        raise ValueError("oracle_dispatch_backslash: bad argument")
    return dict(X=X, kind=kind.value, kl=kl.value, ku=ku.value, info=info.value, AB=AB[:n], ipiv=ipiv[:n])


def detect_bandwidth_cm(Acm: np.ndarray) -> tuple[int, int]:
    """(kl, ku) of the n x n matrix stored COLUMN-major: ``Acm`` has shape (n, lda) and
    ``Acm[j, i]`` is element (i, j) (the row-major array of the transpose)."""
    Acm, n, lda = _dense(Acm)
    kl, ku = ctypes.c_int(), ctypes.c_int()
    rc = _load().oracle_detect_bandwidth_cm(_dptr(Acm), n, max(lda, 1), ctypes.byref(kl), ctypes.byref(ku))
    if rc != 0:
        raise ValueError("oracle_detect_bandwidth_cm: bad argument")
    return kl.value, ku.value


def dense_to_band_cm(Acm: np.ndarray, kl: int, ku: int, ldab: int | None = None) -> np.ndarray:
    """Band storage (n, ldab) of the matrix stored column-major in ``Acm`` (as detect_bandwidth_cm)."""
    Acm, n, lda = _dense(Acm)
    ldab = ldab_for(kl, ku) if ldab is None else ldab
    AB = np.empty((n, ldab), dtype=np.float64)
    rc = _load().oracle_dense_to_band_cm(_dptr(Acm), n, max(lda, 1), kl, ku, _dptr(AB), ldab)
    if rc != 0:
        raise ValueError("oracle_dense_to_band_cm: bad argument")
    return AB
