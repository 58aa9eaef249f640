"""GPU parity of the triangular and diagonal branches of the backslash dispatch (Listing 1)
and of dispatch_backslash as a whole, through the C ABI, against the CPU oracle on the
same seeded inputs: kinds, bandwidths and info exactly, solutions bit for bit (NaN
positions where a solution overflows)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import DEV
from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300.workloads import make_dense

pytestmark = pytest.mark.gpu


def assert_same_solution(got, ref):
    nan_g, nan_r = np.isnan(got), np.isnan(ref)
    assert np.array_equal(nan_g, nan_r)
    if not np.array_equal(got[~nan_g].view(np.int64), ref[~nan_r].view(np.int64)):
        d = np.argwhere(got.view(np.int64) != ref.view(np.int64))[0]
        raise AssertionError(f"solution not bit-identical first at {tuple(d)}: {got[tuple(d)]!r} vs {ref[tuple(d)]!r}")


def triangle(n, k, lower, seed, boost=2.0, dist="normal", pad=5):
    return make_dense(n, k if lower else 0, 0 if lower else k, dist=dist, diag_boost=boost, seed=seed,
                      lda=n + pad).numpy()


def trsv_gpu(A, lower, k, B):
    n, lda = A.shape
    nrhs, ldb = B.shape
    Ad = torch.from_numpy(np.ascontiguousarray(A)).to(DEV)
    Bd = torch.from_numpy(np.ascontiguousarray(B)).to(DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc = bandlu.trsv_band(1 if lower else 0, n, k, Ad, lda, Bd, ldb, nrhs, info)
    torch.cuda.synchronize()
    assert rc == 0, rc
    return Bd.cpu().numpy(), int(info.item())


# register windows of 1, 2, 4, 8 and 16 registers per lane (k+1 <= 512), and the generic kernel
CASES = [(1, 0, 1), (2, 1, 1), (17, 3, 3), (300, 0, 1), (512, 3, 2), (1000, 16, 4), (700, 31, 1), (700, 32, 1),
         (600, 63, 2), (500, 100, 1), (400, 200, 1), (600, 300, 1), (1300, 511, 1), (1200, 600, 1), (300, 299, 1)]


@pytest.mark.parametrize("lower", [True, False])
@pytest.mark.parametrize("n,k,nrhs", CASES)
def test_trsv_band_matches_oracle(n, k, nrhs, lower):
    A = triangle(n, k, lower, seed=5 * n + k + lower)
    B = np.random.default_rng(n + k).standard_normal((nrhs, n + 3))  # ldb = n + 3
    B[:, :2] = 0.0                                                    # the zero skips
    B[:, n - 2:n] = 0.0
    ref, rinfo = oracle.tbsv_dense(A, lower, k, B)
    got, info = trsv_gpu(A, lower, k, B)
    assert info == rinfo == 0
    assert_same_solution(got, ref)


@pytest.mark.parametrize("lower", [True, False])
def test_trsv_band_without_boost_and_singular(lower):
    n, k = 3000, 8
    A = triangle(n, k, lower, seed=31, boost=0.0)                     # growth: infinities, NaNs
    B = np.random.default_rng(1).standard_normal((2, n))
    ref, rinfo = oracle.tbsv_dense(A, lower, k, B)
    got, info = trsv_gpu(A, lower, k, B)
    assert info == rinfo == 0
    assert_same_solution(got, ref)
    A[1234, 1234] = 0.0
    A[2000, 2000] = -0.0
    got, info = trsv_gpu(A, lower, k, B)
    assert info == 1235 and np.array_equal(got, B)


def test_diag_solve_matches_oracle():
    rng = np.random.default_rng(6)
    n, lda = 5000, 5003
    A = np.zeros((n, lda))
    A[np.arange(n), np.arange(n)] = rng.standard_normal(n) * np.exp(rng.uniform(-20, 20, n))
    B = rng.standard_normal((3, n + 1))
    B[0, :10] = 0.0
    Ad, Bd = torch.from_numpy(A).to(DEV), torch.from_numpy(B).to(DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    assert bandlu.diag_solve(n, Ad, lda, Bd, n + 1, 3, info) == 0
    torch.cuda.synchronize()
    ref, rinfo = oracle.diag_solve(A, B)
    assert int(info.item()) == rinfo == 0
    assert_same_solution(Bd.cpu().numpy(), ref)
    A[4321, 4321] = 0.0
    Ad, Bd = torch.from_numpy(A).to(DEV), torch.from_numpy(B).to(DEV)
    assert bandlu.diag_solve(n, Ad, lda, Bd, n + 1, 3, info) == 0
    torch.cuda.synchronize()
    assert int(info.item()) == 4322 and np.array_equal(Bd.cpu().numpy(), B)


def run_backslash(A, B, ldab):
    n, lda = A.shape
    nrhs, ldb = B.shape
    Ad = torch.from_numpy(np.ascontiguousarray(A)).to(DEV)
    Bd = torch.from_numpy(np.ascontiguousarray(B)).to(DEV)
    AB = torch.zeros((max(n, 1), ldab), dtype=torch.float64, device=DEV)
    ipiv = torch.zeros(max(n, 1), dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, kind, kl, ku = bandlu.dispatch_backslash(Ad, n, max(lda, 1), Bd, ldb, nrhs, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    return rc, kind, kl, ku, Bd.cpu().numpy(), int(info.item())


@pytest.mark.parametrize("n,kl,ku,ldab", [(0, 0, 0, 1), (1, 0, 0, 1), (4000, 0, 0, 1), (4000, 9, 0, 1),
                                          (4000, 0, 40, 1), (600, 599, 0, 1), (600, 0, 599, 1),
                                          (4096, 16, 16, 49), (2000, 3, 2, 9), (2000, 3, 2, 8),
                                          (300, 299, 299, 900)])
def test_dispatch_backslash_matches_oracle(n, kl, ku, ldab):
    A = make_dense(n, kl, ku, dist="uniform", diag_boost=2.0 * (kl + ku) + 1.0, seed=n + kl + 2 * ku).numpy()
    B = np.random.default_rng(n).uniform(-1, 1, (2, max(n, 1)))
    rc, kind, gkl, gku, X, info = run_backslash(A, B, ldab)
    r = oracle.dispatch_backslash(A, B, ldab)
    assert (kind, gkl, gku) == (r["kind"], r["kl"], r["ku"]) and (gkl, gku) == (kl, ku)
    if kind == bandlu.KIND_DENSE:
        assert rc == bandlu.BANDLU_NOT_BANDED and np.array_equal(X, B) and info == -5
    else:
        assert rc == 0 and info == r["info"] == 0
        assert_same_solution(X, r["X"])


def test_dispatch_backslash_singular_branches():
    n = 500
    for kl, ku in [(0, 0), (6, 0), (0, 6), (4, 3)]:
        A = make_dense(n, kl, ku, dist="uniform", diag_boost=20.0, seed=kl + 7 * ku).numpy()
        A[321, 321] = 0.0
        if kl and ku:
            A[:, 321] = 0.0                                           # an exactly singular LU
        B = np.random.default_rng(3).standard_normal((1, n))
        rc, kind, _, _, X, info = run_backslash(A, B, 2 * kl + ku + 1)
        r = oracle.dispatch_backslash(A, B, 2 * kl + ku + 1)
        assert rc == 0 and kind == r["kind"] and info == r["info"] == 322
        assert np.array_equal(X, B)
