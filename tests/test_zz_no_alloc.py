"""dispatch_lu_noalloc, the entry point for callers that cannot allocate device
memory (for example when the process's own caching allocator owns all device
memory, or a latency-critical loop forbids allocation calls): through the C ABI
it must give what dispatch_lu gives, on two calls in a row that share its static
scratch array.  Collected last on purpose."""
import numpy as np
import pytest
import torch

from gpu_helpers import DEV, assert_factor_parity
from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300.workloads import make_dense

pytestmark = pytest.mark.gpu


def run(fn, A: torch.Tensor, ldab: int):
    n = A.shape[0]
    AB = torch.full((n, ldab), -3.0, dtype=torch.float64, device=DEV)
    ipiv = torch.full((n,), -1, dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, kl, ku = fn(A, n, n, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    return rc, kl, ku, AB.cpu().numpy(), ipiv.cpu().numpy(), int(info.item())


def test_noalloc_matches_dispatch_lu_on_two_calls_in_a_row():
    # the first call leaves a wider band in the shared scratch than the second needs
    cases = [(make_dense(2048, 20, 9, dist="uniform", seed=71), 2 * 20 + 9 + 1),
             (make_dense(4096, 16, 16, dist="uniform", seed=1002), 49)]
    for A, ldab in cases:
        Ad = A.to(DEV)
        ref = run(bandlu.dispatch_lu, Ad, ldab)
        got = run(bandlu.dispatch_lu_noalloc, Ad, ldab)
        assert got[:3] == ref[:3] and got[0] == 0
        assert_factor_parity(got[3], got[4], got[5], ref[3], ref[4], ref[5])


def test_noalloc_declines_like_dispatch_lu():
    A = make_dense(1000, 3, 3, dist="uniform", seed=5)
    A[999, 0] = 1e-3
    Ad = A.to(DEV)
    ref = run(bandlu.dispatch_lu, Ad, 10)
    got = run(bandlu.dispatch_lu_noalloc, Ad, 10)
    assert got[:3] == ref[:3] == (bandlu.BANDLU_NOT_BANDED, 999, 3)
    assert np.all(got[3] == -3.0) and np.all(got[4] == -1) and got[5] == -5


def test_noalloc_wide_band_matches_dispatch_lu():
    # wide band: dispatch_lu takes the multi-CTA kernel, the allocation-free entry
    # point the single-CTA one; both reproduce the unblocked elimination exactly
    A = make_dense(1200, 40, 30, dist="normal", seed=91)
    Ad = A.to(DEV)
    ref = run(bandlu.dispatch_lu, Ad, 111)
    got = run(bandlu.dispatch_lu_noalloc, Ad, 111)
    assert got[:3] == ref[:3] == (0, 40, 30)
    assert_factor_parity(got[3], got[4], got[5], ref[3], ref[4], ref[5])


def _loaded_cudart():
    """The CUDA runtime library torch loaded in this process (its default memory pool is the
    device's, shared with every runtime in the process)."""
    import ctypes
    torch.cuda.init()
    with open("/proc/self/maps") as f:
        paths = {ln.split()[-1] for ln in f if "libcudart" in ln and ln.split()[-1].startswith("/")}
    if not paths:
        pytest.skip("no dynamically loaded CUDA runtime to query the memory pool with")
    rt = ctypes.CDLL(sorted(paths)[0])
    return rt


def _pool_used_high(rt, pool) -> int:
    import ctypes
    v = ctypes.c_uint64(0)
    assert rt.cudaMemPoolGetAttribute(pool, 0x8, ctypes.byref(v)) == 0  # cudaMemPoolAttrUsedMemHigh
    return v.value


def _pool_reset_high(rt, pool) -> None:
    import ctypes
    z = ctypes.c_uint64(0)
    assert rt.cudaMemPoolSetAttribute(pool, 0x8, ctypes.byref(z)) == 0


def test_noalloc_takes_nothing_from_the_stream_ordered_pool():
    """The property the entry point exists for: its calls leave the device's default
    memory pool untouched (high-water mark reset before, read after), while dispatch_lu's
    8 bytes of scratch do register there -- which shows the probe sees such allocations."""
    import ctypes
    rt = _loaded_cudart()
    pool = ctypes.c_void_p()
    assert rt.cudaDeviceGetDefaultMemPool(ctypes.byref(pool), 0) == 0
    cases = [(make_dense(1500, 12, 7, dist="uniform", seed=33), 2 * 12 + 7 + 1),
             (make_dense(1200, 40, 30, dist="normal", seed=91), 111)]   # the wide band too
    dev_cases = [(A.to(DEV), ldab) for A, ldab in cases]
    torch.cuda.synchronize()
    for Ad, ldab in dev_cases:
        run(bandlu.dispatch_lu_noalloc, Ad, ldab)          # set-up of this device done
        torch.cuda.synchronize()
        assert rt.cudaMemPoolTrimTo(pool, ctypes.c_size_t(0)) == 0
        _pool_reset_high(rt, pool)
        assert _pool_used_high(rt, pool) == 0
        got = run(bandlu.dispatch_lu_noalloc, Ad, ldab)
        assert got[0] == 0
        assert _pool_used_high(rt, pool) == 0
    # the positive control: dispatch_lu's stream-ordered scratch shows up in the pool
    _pool_reset_high(rt, pool)
    run(bandlu.dispatch_lu, dev_cases[0][0], dev_cases[0][1])
    assert _pool_used_high(rt, pool) > 0


def test_noalloc_matches_the_oracle():
    import oracle
    A = make_dense(3000, 9, 14, dist="uniform", seed=57)
    ldab = 2 * 9 + 14 + 1
    got = run(bandlu.dispatch_lu_noalloc, A.to(DEV), ldab)
    ref = oracle.dispatch_lu(A.numpy(), ldab)
    assert got[:3] == (ref["status"], ref["kl"], ref["ku"]) == (0, 9, 14)
    assert_factor_parity(got[3], got[4], got[5], ref["AB"], ref["ipiv"], ref["info"])
