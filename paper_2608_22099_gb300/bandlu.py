"""Thin ctypes binding of the C ABI in include/bandlu.h (argument marshalling only).

Every function has the C name and the C argument order.  Pointer arguments take
a torch tensor (its data_ptr is passed) or a raw integer address; ``stream``
takes a torch.cuda.Stream, a raw cudaStream_t integer, or None for torch's
current stream.  All arithmetic runs in the CUDA library; there is no CPU or
PyTorch fallback: if the library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

BANDLU_OK = 0
BANDLU_NOT_BANDED = 1
BANDLU_ERR_CUDA = 1000
BANDLU_ERR_TIMEOUT = 1001
BANDLU_ERR_SCRATCH = 1002

_lock = threading.Lock()
_lib = None


class BandLUError(RuntimeError):
    pass


def library_path() -> str:
    return _build.LIB


def load():
    """Load libbandlu.so (building it first if the sources are newer)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        # BANDLU_CHECKED=1 selects the checked build (bounded inter-warp waits) for
        # development runs; the default is the production library.
        checked = os.environ.get("BANDLU_CHECKED", "") == "1"
        # BANDLU_TRACE=1 selects the traced build (timeline of the wide-band chain kernel)
        trace = not checked and os.environ.get("BANDLU_TRACE", "") == "1"
        path = _build.CHECKED_LIB if checked else (_build.TRACE_LIB if trace else _build.LIB)
        if not _build.up_to_date(path):
            try:
                path = _build.build(checked=checked, trace=trace)
            except Exception as e:  # noqa: BLE001 - re-raised with context
                raise BandLUError(f"the CUDA library could not be built: {e}") from e
        if not os.path.exists(path):
            raise BandLUError(f"CUDA library missing at {path}")
        lib = ctypes.CDLL(path)
        vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        lib.detect_bandwidth.argtypes = [vp, i64, i64, vp, vp, vp]
        lib.dense_to_band.argtypes = [vp, i64, i64, i32, i32, vp, i64, vp]
        lib.gbtrf.argtypes = [i64, i32, i32, vp, i64, vp, vp, vp]
        lib.dispatch_lu.argtypes = [vp, i64, i64, vp, i64, vp, vp, vp, vp, vp]
        lib.dispatch_lu_noalloc.argtypes = [vp, i64, i64, vp, i64, vp, vp, vp, vp, vp]
        lib.dispatch_lu_batched.argtypes = [vp, i64, i64, i64, i64, vp, i64, i64, vp, i64, vp, vp, vp, vp, vp]
        lib.gbtrs.argtypes = [i64, i32, i32, i64, vp, i64, vp, vp, i64, vp]
        lib.dispatch_solve.argtypes = [vp, i64, i64, vp, i64, i64, vp, i64, vp, vp, vp, vp, vp]
        lib.detect_bandwidth_cm.argtypes = [vp, i64, i64, vp, vp, vp]
        lib.dense_to_band_cm.argtypes = [vp, i64, i64, i32, i32, vp, i64, vp]
        lib.dispatch_lu_cm.argtypes = [vp, i64, i64, vp, i64, vp, vp, vp, vp, vp]
        lib.dispatch_lu_async.argtypes = [vp, i64, i64, vp, i64, vp, vp, vp, vp, vp, vp]
        lib.trsv_band.argtypes = [i32, i64, i32, vp, i64, vp, i64, i64, vp, vp]
        lib.diag_solve.argtypes = [i64, vp, i64, vp, i64, i64, vp, vp]
        lib.bandlu_classify.argtypes = [i64, i32, i32, i64]
        lib.dispatch_backslash.argtypes = [vp, i64, i64, vp, i64, i64, vp, i64, vp, vp, vp, vp, vp, vp]
        for f in ("detect_bandwidth", "dense_to_band", "gbtrf", "gbtrs", "dispatch_lu", "dispatch_solve",
                  "dispatch_lu_batched", "dispatch_lu_noalloc", "dispatch_lu_async", "trsv_band",
                  "detect_bandwidth_cm", "dense_to_band_cm", "dispatch_lu_cm", "diag_solve", "bandlu_classify",
                  "dispatch_backslash"):
            getattr(lib, f).restype = ctypes.c_int
        lib.bandlu_trace_capacity.argtypes = []
        lib.bandlu_trace_capacity.restype = ctypes.c_int
        lib.bandlu_trace_read.argtypes = [vp, i64]
        lib.bandlu_trace_read.restype = ctypes.c_int
        lib.bandlu_trace_clear.argtypes = []
        lib.bandlu_trace_clear.restype = ctypes.c_int
        lib.bandlu_selftest_rcp_host.argtypes = [vp, vp, i64]
        lib.bandlu_selftest_rcp_host.restype = None
        lib.bandlu_selftest_rcp_device.argtypes = [vp, vp, i64, i32, vp]
        lib.bandlu_selftest_rcp_device.restype = ctypes.c_int
        lib.bandlu_selftest_div_host.argtypes = [vp, vp, vp, i64]
        lib.bandlu_selftest_div_host.restype = None
        lib.bandlu_selftest_div_nz_host.argtypes = [vp, vp, vp, i64]
        lib.bandlu_selftest_div_nz_host.restype = None
        lib.bandlu_selftest_div_device.argtypes = [vp, vp, vp, i64, i32, vp]
        lib.bandlu_selftest_div_device.restype = ctypes.c_int
        lib.bandlu_peak_dfma.argtypes = [vp, i32, i32, i32, i32, vp]
        lib.bandlu_peak_dmma.argtypes = [i32, vp, i32, i32, i32, i32, vp]
        lib.bandlu_peak_hbm_read.argtypes = [vp, i64, vp, i32, vp]
        lib.bandlu_peak_warp_costs.argtypes = [i32, vp, vp, i32, i32, vp]
        for f in ("bandlu_peak_dfma", "bandlu_peak_dmma", "bandlu_peak_hbm_read", "bandlu_peak_warp_costs"):
            getattr(lib, f).restype = ctypes.c_int
        lib.bandlu_version.restype = ctypes.c_char_p
        lib.bandlu_version.argtypes = []
        _lib = lib
        return lib


def _ptr(x) -> int:
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _stream(s) -> int:
    if s is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(s, int):
        return s
    return int(s.cuda_stream)


def version() -> str:
    return load().bandlu_version().decode()


def detect_bandwidth(A, n: int, lda: int, d_kl, d_ku, stream=None) -> int:
    return load().detect_bandwidth(_ptr(A), n, lda, _ptr(d_kl), _ptr(d_ku), _stream(stream))


def dense_to_band(A, lda: int, n: int, kl: int, ku: int, AB, ldab: int, stream=None) -> int:
    return load().dense_to_band(_ptr(A), lda, n, kl, ku, _ptr(AB), ldab, _stream(stream))


def gbtrf(n: int, kl: int, ku: int, AB, ldab: int, ipiv, d_info, stream=None) -> int:
    return load().gbtrf(n, kl, ku, _ptr(AB), ldab, _ptr(ipiv), _ptr(d_info), _stream(stream))


def dispatch_lu(A, n: int, lda: int, AB, ldab: int, ipiv, d_info, stream=None) -> tuple[int, int, int]:
    """Returns (status, kl, ku); kl and ku are the host outputs of the C call."""
    kl, ku = ctypes.c_int(-1), ctypes.c_int(-1)
    rc = load().dispatch_lu(_ptr(A), n, lda, _ptr(AB), ldab, _ptr(ipiv), ctypes.addressof(kl),
                            ctypes.addressof(ku), _ptr(d_info), _stream(stream))
    return rc, kl.value, ku.value


def detect_bandwidth_cm(A, n: int, lda: int, d_kl, d_ku, stream=None) -> int:
    """detect_bandwidth for a column-major A (element (i, j) at A[i + j*lda])."""
    return load().detect_bandwidth_cm(_ptr(A), n, lda, _ptr(d_kl), _ptr(d_ku), _stream(stream))


def dense_to_band_cm(A, lda: int, n: int, kl: int, ku: int, AB, ldab: int, stream=None) -> int:
    """dense_to_band for a column-major A."""
    return load().dense_to_band_cm(_ptr(A), lda, n, kl, ku, _ptr(AB), ldab, _stream(stream))


def dispatch_lu_cm(A, n: int, lda: int, AB, ldab: int, ipiv, d_info, stream=None) -> tuple[int, int, int]:
    """dispatch_lu for a column-major A.  Returns (status, kl, ku)."""
    kl, ku = ctypes.c_int(-1), ctypes.c_int(-1)
    rc = load().dispatch_lu_cm(_ptr(A), n, lda, _ptr(AB), ldab, _ptr(ipiv), ctypes.addressof(kl),
                               ctypes.addressof(ku), _ptr(d_info), _stream(stream))
    return rc, kl.value, ku.value


def dispatch_lu_async(A, n: int, lda: int, AB, ldab: int, ipiv, d_kl, d_ku, d_status, d_info, stream=None) -> int:
    """dispatch_lu with the decision on the device: no host synchronisation; outputs in device memory."""
    return load().dispatch_lu_async(_ptr(A), n, lda, _ptr(AB), ldab, _ptr(ipiv), _ptr(d_kl), _ptr(d_ku),
                                    _ptr(d_status), _ptr(d_info), _stream(stream))


def gbtrs(n: int, kl: int, ku: int, nrhs: int, AB, ldab: int, ipiv, B, ldb: int, stream=None) -> int:
    return load().gbtrs(n, kl, ku, nrhs, _ptr(AB), ldab, _ptr(ipiv), _ptr(B), ldb, _stream(stream))


def dispatch_solve(A, n: int, lda: int, B, ldb: int, nrhs: int, AB, ldab: int, ipiv, d_info,
                   stream=None) -> tuple[int, int, int]:
    """Returns (status, kl, ku); kl and ku are the host outputs of the C call."""
    kl, ku = ctypes.c_int(-1), ctypes.c_int(-1)
    rc = load().dispatch_solve(_ptr(A), n, lda, _ptr(B), ldb, nrhs, _ptr(AB), ldab, _ptr(ipiv),
                               ctypes.addressof(kl), ctypes.addressof(ku), _ptr(d_info), _stream(stream))
    return rc, kl.value, ku.value


# Branches of the backslash dispatch (BANDLU_KIND_* of bandlu.h).
KIND_DIAGONAL, KIND_LOWER, KIND_UPPER, KIND_BANDED, KIND_DENSE = 1, 2, 3, 4, 5


def trsv_band(lower: int, n: int, k: int, A, lda: int, B, ldb: int, nrhs: int, d_info, stream=None) -> int:
    return load().trsv_band(lower, n, k, _ptr(A), lda, _ptr(B), ldb, nrhs, _ptr(d_info), _stream(stream))


def diag_solve(n: int, A, lda: int, B, ldb: int, nrhs: int, d_info, stream=None) -> int:
    return load().diag_solve(n, _ptr(A), lda, _ptr(B), ldb, nrhs, _ptr(d_info), _stream(stream))


def bandlu_classify(n: int, kl: int, ku: int, ldab: int) -> int:
    """The branch of the backslash dispatch for bandwidths (kl, ku) (host logic, no GPU work)."""
    return load().bandlu_classify(n, kl, ku, ldab)


def dispatch_backslash(A, n: int, lda: int, B, ldb: int, nrhs: int, AB, ldab: int, ipiv, d_info,
                       stream=None) -> tuple[int, int, int, int]:
    """Returns (status, kind, kl, ku); kind, kl and ku are the host outputs of the C call."""
    kl, ku, kind = ctypes.c_int(-1), ctypes.c_int(-1), ctypes.c_int(-1)
    rc = load().dispatch_backslash(_ptr(A), n, lda, _ptr(B), ldb, nrhs, _ptr(AB), ldab, _ptr(ipiv),
                                   ctypes.addressof(kl), ctypes.addressof(ku), ctypes.addressof(kind),
                                   _ptr(d_info), _stream(stream))
    return rc, kind.value, kl.value, ku.value


def dispatch_lu_noalloc(A, n: int, lda: int, AB, ldab: int, ipiv, d_info, stream=None) -> tuple[int, int, int]:
    """dispatch_lu without device allocation (scratch in a static device array).
    Returns (status, kl, ku)."""
    kl, ku = ctypes.c_int(-1), ctypes.c_int(-1)
    rc = load().dispatch_lu_noalloc(_ptr(A), n, lda, _ptr(AB), ldab, _ptr(ipiv), ctypes.addressof(kl),
                                    ctypes.addressof(ku), _ptr(d_info), _stream(stream))
    return rc, kl.value, ku.value


def dispatch_lu_batched(A, n: int, lda: int, strideA: int, batch: int, AB, ldab: int, strideAB: int, ipiv,
                        strideP: int, d_kl, d_ku, d_info, d_status, stream=None) -> int:
    return load().dispatch_lu_batched(_ptr(A), n, lda, strideA, batch, _ptr(AB), ldab, strideAB, _ptr(ipiv),
                                      strideP, _ptr(d_kl), _ptr(d_ku), _ptr(d_info), _ptr(d_status),
                                      _stream(stream))


def bandlu_trace_capacity() -> int:
    """Panels the traced build records per role (0 in the production build)."""
    return load().bandlu_trace_capacity()


def bandlu_trace_read(host, count: int) -> int:
    """Copies the first `count` words of the chain kernel's timeline to `host` (host buffer)."""
    return load().bandlu_trace_read(_ptr_host(host), count)


def bandlu_trace_clear() -> int:
    """Zeroes the timeline (traced build)."""
    return load().bandlu_trace_clear()


def bandlu_selftest_rcp_host(x, y, n: int) -> None:
    """Self-test hook: the library's reciprocal on the host (x, y: host buffers of n doubles)."""
    load().bandlu_selftest_rcp_host(_ptr_host(x), _ptr_host(y), n)


def bandlu_selftest_rcp_device(x, y, n: int, use_division: int, stream=None) -> int:
    """Self-test hook: the library's reciprocal (or plain division) on the device."""
    return load().bandlu_selftest_rcp_device(_ptr(x), _ptr(y), n, use_division, _stream(stream))


def bandlu_selftest_div_host(x, d, q, n: int) -> None:
    """Self-test hook: the library's known-divisor division on the host (host buffers of n doubles)."""
    load().bandlu_selftest_div_host(_ptr_host(x), _ptr_host(d), _ptr_host(q), n)


def bandlu_selftest_div_nz_host(x, d, q, n: int) -> None:
    """Self-test hook: the back substitution's quotient with its zero test, on the host."""
    load().bandlu_selftest_div_nz_host(_ptr_host(x), _ptr_host(d), _ptr_host(q), n)


def bandlu_selftest_div_device(x, d, q, n: int, use_division: int, stream=None) -> int:
    """Self-test hook: the library's known-divisor division (or plain division) on the device."""
    return load().bandlu_selftest_div_device(_ptr(x), _ptr(d), _ptr(q), n, use_division, _stream(stream))


def bandlu_peak_dfma(d_sink, blocks: int, threads: int, chains: int, iters: int, stream=None) -> int:
    """Microbenchmark launch: 2*blocks*threads*chains*iters FP64 flops of independent FMA chains."""
    return load().bandlu_peak_dfma(_ptr(d_sink), blocks, threads, chains, iters, _stream(stream))


def bandlu_peak_dmma(shape: int, d_sink, blocks: int, warps: int, chains: int, iters: int, stream=None) -> int:
    """Microbenchmark launch: FP64 mma.sync (shape 0 m8n8k4, 1 m16n8k16), chains accumulators per warp."""
    return load().bandlu_peak_dmma(shape, _ptr(d_sink), blocks, warps, chains, iters, _stream(stream))


def bandlu_peak_warp_costs(op: int, d_clk, d_sink, warps: int, iters: int, stream=None) -> int:
    """Microbenchmark launch: one block of `warps` warps, 16 * iters instances of operation `op`
    (0..7, see include/bandlu_peaks.h); d_clk receives thread 0's elapsed clock cycles."""
    return load().bandlu_peak_warp_costs(op, _ptr(d_clk), _ptr(d_sink), warps, iters, _stream(stream))


def bandlu_peak_hbm_read(d_buf, nbytes: int, d_sink, blocks: int, stream=None) -> int:
    """Microbenchmark launch: one read-only pass over nbytes of device memory."""
    return load().bandlu_peak_hbm_read(_ptr(d_buf), nbytes, _ptr(d_sink), blocks, _stream(stream))


def _ptr_host(x) -> int:
    if isinstance(x, int):
        return x
    if hasattr(x, "ctypes"):
        return int(x.ctypes.data)
    return int(x.data_ptr())


def check(rc: int, what: str = "call") -> int:
    """Raise BandLUError for an error status (negative or >= BANDLU_ERR_CUDA)."""
    if rc < 0:
        raise BandLUError(f"{what}: invalid argument {-rc}")
    if rc >= BANDLU_ERR_CUDA:
        raise BandLUError(f"{what}: status {rc}")
    return rc
