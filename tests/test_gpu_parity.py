"""GPU parity: every entry point, called through the C ABI, against the CPU oracle on
the same seeded inputs.  Integers (kl, ku, ipiv, info, status) must match bit for
bit; factors within 1e-12 relative in the inf-norm (the bar), and the kernels are
also checked to be bit-identical to the oracle, which they are designed to be."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import DEV, assert_factor_parity, convert_gpu, detect_gpu, gbtrf_gpu
from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300.workloads import make_dense

pytestmark = pytest.mark.gpu


def banded(n, kl, ku, seed, boost=0.0, dist="uniform", lda=None):
    return make_dense(n, kl, ku, dist=dist, diag_boost=boost, seed=seed, lda=lda)


# --------------------------------------------------------------------------------------------
# detect_bandwidth
# --------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,kl,ku", [(1, 0, 0), (2, 1, 0), (3, 0, 2), (17, 3, 5), (64, 16, 16), (255, 31, 2),
                                     (256, 2, 2), (512, 3, 3), (1000, 7, 90), (1023, 1, 1), (2049, 5, 6),
                                     (4096, 16, 16), (5000, 0, 0)])
def test_detect_matches_oracle(n, kl, ku):
    A = banded(n, kl, ku, seed=n + 3 * kl + ku)
    expect = oracle.detect_bandwidth(A.numpy())
    assert expect == (kl, ku)
    assert detect_gpu(A.to(DEV)) == expect


def test_detect_special_cases():
    n = 300
    z = torch.zeros((n, n), dtype=torch.float64)
    assert detect_gpu(z.to(DEV)) == (0, 0)
    full = torch.rand((n, n), dtype=torch.float64, generator=torch.Generator().manual_seed(1)) + 0.5
    assert detect_gpu(full.to(DEV)) == (n - 1, n - 1)
    for (i, j), expect in [((n - 1, 0), (n - 1, 0)), ((0, n - 1), (0, n - 1)), ((150, 149), (1, 0))]:
        s = z.clone(); s[i, j] = 1e-3
        assert detect_gpu(s.to(DEV)) == expect
    neg0 = z.clone(); neg0[n - 1, 0] = -0.0
    assert detect_gpu(neg0.to(DEV)) == (0, 0)
    for v in (float("nan"), float("inf"), 5e-324):
        s = z.clone(); s[n - 5, 2] = v
        assert detect_gpu(s.to(DEV)) == (n - 7, 0)


@pytest.mark.parametrize("n", [1025, 2049])
def test_detect_contiguous_odd_rows_ignore_padding(n):
    """Rows of odd length n stored with lda = n+1 form one contiguous run of 16-byte vectors:
    the padding column (garbage here, NaN and ones) is never counted, and a stray entry in the
    matrix's very last element or first column of the last row is found."""
    lda = n + 1
    A = banded(n, 3, 5, seed=n, lda=lda)
    A[:, n] = float("nan")
    A[::2, n] = 1.0
    assert detect_gpu(A.to(DEV), n, lda) == (3, 5)
    B = A.clone()
    B[n - 1, n - 1] = 0.0
    B[0, n - 1] = 2.0                      # ku = n-1
    assert detect_gpu(B.to(DEV), n, lda) == (3, n - 1)
    C = A.clone()
    C[n - 1, 0] = -1.0                     # kl = n-1
    assert detect_gpu(C.to(DEV), n, lda) == (n - 1, 5)


@pytest.mark.parametrize("n,lda", [(100, 101), (99, 100), (99, 99), (1000, 1003), (2048, 2050)])
def test_detect_lda_padding_and_scalar_path(n, lda):
    A = banded(n, 4, 9, seed=n, lda=lda)
    A[:, n:] = 7.0                      # padding must be ignored
    assert detect_gpu(A.to(DEV), n, lda) == (4, 9)


def test_detect_misaligned_base():
    n, lda = 400, 402
    buf = torch.zeros(n * lda + 1, dtype=torch.float64)
    M = buf[1:].view(n, lda)            # 8-byte but not 16-byte aligned
    M.copy_(banded(n, 3, 11, seed=9, lda=lda))
    Md = torch.zeros(n * lda + 1, dtype=torch.float64, device=DEV)
    Md[1:].copy_(M.reshape(-1))
    out = torch.zeros(2, dtype=torch.int32, device=DEV)
    assert bandlu.detect_bandwidth(Md.data_ptr() + 8, n, lda, out, out.data_ptr() + 4) == 0
    torch.cuda.synchronize()
    assert out.tolist() == [3, 11]


def test_detect_separate_output_pointers():
    A = banded(500, 6, 2, seed=2).to(DEV)
    kl = torch.full((1,), 99, dtype=torch.int32, device=DEV)
    ku = torch.full((1,), 99, dtype=torch.int32, device=DEV)
    assert bandlu.detect_bandwidth(A, 500, 500, kl, ku) == 0
    torch.cuda.synchronize()
    assert (kl.item(), ku.item()) == (6, 2)


# --------------------------------------------------------------------------------------------
# dense_to_band
# --------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,kl,ku,extra", [(1, 0, 0, 0), (5, 1, 1, 0), (40, 7, 0, 0), (40, 0, 7, 2),
                                           (512, 3, 3, 0), (1000, 16, 16, 3), (300, 100, 150, 0),
                                           (2000, 1000, 1500, 0), (33, 32, 32, 0)])
def test_convert_matches_oracle_bitwise(n, kl, ku, extra):
    A = banded(n, kl, ku, seed=n + kl, lda=n + (n % 3))
    ldab = 2 * kl + ku + 1 + extra
    ref = oracle.dense_to_band(A.numpy(), kl, ku, ldab)
    got = convert_gpu(A.to(DEV), kl, ku, ldab).cpu().numpy()
    assert np.array_equal(got.view(np.int64), ref.view(np.int64))


def test_convert_reads_only_the_band():
    n, kl, ku = 200, 5, 4
    A = banded(n, kl, ku, seed=3)
    # entries outside the requested band are garbage; they must not reach AB
    noisy = A.clone()
    mask = torch.ones((n, n), dtype=torch.bool)
    for d in range(-kl, ku + 1):
        mask.diagonal(d).fill_(False)
    noisy[mask] = float("nan")
    ref = oracle.dense_to_band(A.numpy(), kl, ku)
    got = convert_gpu(noisy.to(DEV), kl, ku, 2 * kl + ku + 1).cpu().numpy()
    assert np.array_equal(got.view(np.int64), ref.view(np.int64))


# --------------------------------------------------------------------------------------------
# gbtrf
# --------------------------------------------------------------------------------------------

GBTRF_CASES = [
    (1, 0, 0), (2, 1, 1), (3, 2, 0), (5, 0, 4), (8, 1, 1), (17, 3, 5), (64, 16, 16), (100, 27, 3),
    (100, 28, 3), (257, 8, 64), (300, 2, 2), (512, 3, 3), (700, 0, 12), (700, 12, 0), (1000, 31, 31),
    (600, 40, 40), (130, 1, 100), (96, 5, 90), (2000, 16, 16),
]


@pytest.mark.parametrize("n,kl,ku", GBTRF_CASES)
@pytest.mark.parametrize("dist", ["uniform", "normal"])
def test_gbtrf_matches_oracle(n, kl, ku, dist):
    A = banded(n, kl, ku, seed=7 * n + kl + ku, dist=dist).numpy()
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    got = gbtrf_gpu(AB, kl, ku)
    assert_factor_parity(*got, ref[0], ref[1], ref[2])
    assert oracle.backward_error(A, got[0], got[1], kl, ku) <= 10.0


@pytest.mark.parametrize("kl,ku", [(1, 1), (4, 3), (30, 10)])
def test_gbtrf_zero_pivots_and_zero_columns(kl, ku):
    n = 150
    A = banded(n, kl, ku, seed=kl, boost=0.5).numpy()
    A[:, 20] = 0.0                      # exact zero column -> info = 21
    A[:, 77] = 0.0
    A[40, :] = 0.0                      # exact zero row -> a zero pivot later
    A[90:93, 91] = -0.0
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    assert ref[2] == 21
    got = gbtrf_gpu(AB, kl, ku)
    assert_factor_parity(*got, ref[0], ref[1], ref[2])


def test_gbtrf_forced_interchanges_every_column():
    n = 500
    A = np.diag(np.full(n, 1e-3)) + np.diag(np.ones(n - 1), -1) + np.diag(np.full(n - 1, 0.5), 1)
    for kl, ku in [(1, 1), (3, 2)]:
        AB = oracle.dense_to_band(A, kl, ku)
        ref = oracle.gbtrf(AB, kl, ku)
        assert np.array_equal(ref[1][:-1], np.arange(2, n + 1, dtype=np.int32))
        assert_factor_parity(*gbtrf_gpu(AB, kl, ku), ref[0], ref[1], ref[2])


def test_gbtrf_pivot_ties_take_the_first_row():
    n, kl, ku = 64, 3, 2
    A = np.zeros((n, n))
    for i in range(n):
        for j in range(max(0, i - kl), min(n, i + ku + 1)):
            A[i, j] = 1.0 if (i + j) % 2 == 0 else -1.0   # equal magnitudes everywhere
    A += np.diag(np.full(n, 0.0))
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    assert_factor_parity(*gbtrf_gpu(AB, kl, ku), ref[0], ref[1], ref[2])


@pytest.mark.parametrize("n,kl,ku", [(300, 6, 5), (300, 2, 3), (257, 0, 9), (200, 30, 12)])
def test_gbtrf_garbage_in_fill_rows_and_wider_storage(n, kl, ku):
    # fill rows hold garbage (the elimination clears them); rows beyond 2kl+ku hold
    # garbage that no step may touch (the oracle leaves them as they are)
    A = banded(n, kl, ku, seed=5 + kl).numpy()
    ldab = 2 * kl + ku + 1 + 3
    AB = oracle.dense_to_band(A, kl, ku, ldab=ldab)
    AB[:, :kl] = 321.0
    AB[:, 2 * kl + ku + 1:] = -17.25
    ref = oracle.gbtrf(AB, kl, ku)
    assert np.all(ref[0][:, 2 * kl + ku + 1:] == -17.25)
    assert_factor_parity(*gbtrf_gpu(AB, kl, ku), ref[0], ref[1], ref[2])


def test_gbtrf_tridiagonal_closed_form_on_gpu():
    n = 20000
    AB = np.zeros((n, 4)); AB[:, 2] = 2.0; AB[1:, 1] = -1.0; AB[:-1, 3] = -1.0
    ABf, ipiv, info = gbtrf_gpu(AB, 1, 1)
    j = np.arange(n)
    assert info == 0 and np.array_equal(ipiv, (j + 1).astype(np.int32))
    tol = 4 * 2.0 ** -52 * (j + 1)
    assert np.all(np.abs(ABf[:, 2] - (j + 2) / (j + 1)) <= tol * (j + 2) / (j + 1))
    assert abs(np.sum(np.log(ABf[:, 2])) - np.log(n + 1)) < 1e-12 * n


def test_gbtrf_deterministic():
    n, kl, ku = 3000, 16, 16
    AB = oracle.dense_to_band(banded(n, kl, ku, seed=1).numpy(), kl, ku)
    a = gbtrf_gpu(AB, kl, ku)
    b = gbtrf_gpu(AB, kl, ku)
    assert np.array_equal(a[0].view(np.int64), b[0].view(np.int64)) and np.array_equal(a[1], b[1])


def test_gbtrf_empty():
    AB = torch.zeros((1, 1), dtype=torch.float64, device=DEV)
    info = torch.full((1,), 9, dtype=torch.int32, device=DEV)
    ipiv = torch.zeros(1, dtype=torch.int32, device=DEV)
    assert bandlu.gbtrf(0, 0, 0, AB, 1, ipiv, info) == 0
    torch.cuda.synchronize()
    assert info.item() == 0


# --------------------------------------------------------------------------------------------
# wide bands (kl beyond the windowed kernel): the multi-CTA panel/update kernel
# --------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,kl,ku", [(12, 28, 0), (13, 29, 1), (50, 30, 28), (203, 28, 0), (401, 33, 70),
                                     (777, 64, 5), (1030, 100, 100), (2049, 256, 256)])
def test_gbtrf_wide_matches_oracle(n, kl, ku):
    A = banded(n, kl, ku, seed=11 * n + kl + 3 * ku, dist="normal").numpy()
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    got = gbtrf_gpu(AB, kl, ku)
    assert_factor_parity(*got, ref[0], ref[1], ref[2])
    assert oracle.backward_error(A, got[0], got[1], kl, ku) <= 10.0


def test_gbtrf_wide_blocks_share_update_ctas():
    # kv = 700: one panel reaches more column blocks than there are update CTAs,
    # so update CTAs hold two blocks at once.
    n, kl, ku = 2003, 300, 400
    A = banded(n, kl, ku, seed=17, boost=2.0).numpy()
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    assert_factor_parity(*gbtrf_gpu(AB, kl, ku), ref[0], ref[1], ref[2])


@pytest.mark.parametrize("n,kl,ku", [(701, 600, 10), (613, 290, 33)])
def test_gbtrf_wide_several_rows_per_thread(n, kl, ku):
    # kl + 4 panel rows exceed one compute group's 288 threads: 2 (kl = 290) and 3-4 (kl = 600)
    # rows per thread
    A = banded(n, kl, ku, seed=n + kl, dist="normal").numpy()
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    got = gbtrf_gpu(AB, kl, ku)
    assert_factor_parity(*got, ref[0], ref[1], ref[2])
    assert oracle.backward_error(A, got[0], got[1], kl, ku) <= 10.0


def test_gbtrf_wide_zero_pivots_garbage_fill_and_wider_storage():
    n, kl, ku = 500, 40, 31
    A = banded(n, kl, ku, seed=23).numpy()
    A[:, 77] = 0.0
    A[200:240, 200:240] = 0.0
    AB = oracle.dense_to_band(A, kl, ku, ldab=2 * kl + ku + 1 + 5)
    AB[:, :kl] = -9.5
    ref = oracle.gbtrf(AB, kl, ku)
    assert ref[2] > 0
    assert_factor_parity(*gbtrf_gpu(AB, kl, ku), ref[0], ref[1], ref[2])


def test_gbtrf_wide_deterministic():
    n, kl, ku = 1500, 48, 48
    AB = oracle.dense_to_band(banded(n, kl, ku, seed=2).numpy(), kl, ku)
    a = gbtrf_gpu(AB, kl, ku)
    b = gbtrf_gpu(AB, kl, ku)
    assert np.array_equal(a[0].view(np.int64), b[0].view(np.int64)) and np.array_equal(a[1], b[1])


# --------------------------------------------------------------------------------------------
# NaN candidates: the pivot rule of the comparison order (a NaN is kept only as the first
# candidate), in every kernel
# --------------------------------------------------------------------------------------------

def assert_parity_with_nan(AB, ipiv, info, ABr, ipr, infr):
    assert info == infr and np.array_equal(ipiv, ipr)
    nan_g, nan_r = np.isnan(AB), np.isnan(ABr)
    assert np.array_equal(nan_g, nan_r)                  # NaN payloads may differ; positions may not
    assert np.array_equal(AB[~nan_g].view(np.int64), ABr[~nan_r].view(np.int64))


def plant_nans(A, kl, ku):
    n = A.shape[0]
    r0 = max(0, n - 60)
    for (i, j) in ((r0 + 3, r0), (r0 + 1, r0 + 1), (r0 + 9, r0 + 7), (r0 + 12, r0 + 12)):
        if i < n and j < n and -ku <= j - i <= kl and i - j <= kl:
            A[i, j] = np.nan
    return A


@pytest.mark.parametrize("n,kl,ku", [(300, 5, 4), (200, 27, 3), (400, 40, 30), (14, 30, 2)])
def test_gbtrf_nan_candidates(n, kl, ku):
    A = plant_nans(banded(n, kl, ku, seed=n + kl, dist="normal").numpy(), kl, ku)
    AB = oracle.dense_to_band(A, kl, ku)
    ref = oracle.gbtrf(AB, kl, ku)
    assert_parity_with_nan(*gbtrf_gpu(AB, kl, ku), ref[0], ref[1], ref[2])


@pytest.mark.parametrize("n,kl,ku", [(64, 3, 3), (100, 40, 8)])
def test_batched_nan_candidates(n, kl, ku):
    batch = 6
    A = torch.stack([torch.from_numpy(plant_nans(banded(n, kl, ku, seed=b).numpy(), kl, ku)) for b in range(batch)])
    ldab = 2 * kl + ku + 1
    got = run_batched(A, ldab)
    ref = oracle.dispatch_lu_batched(A.numpy(), ldab)
    for key in ("kl", "ku", "status", "info"):
        assert np.array_equal(got[key], ref[key]), key
    for b in range(batch):
        assert_parity_with_nan(got["AB"][b], got["ipiv"][b], int(got["info"][b]), ref["AB"][b], ref["ipiv"][b],
                               int(ref["info"][b]))


# --------------------------------------------------------------------------------------------
# gbtrs (the solve after the factorisation) and dispatch_solve
# --------------------------------------------------------------------------------------------

def gbtrs_gpu(ABf, ipiv, kl, ku, B):
    n, ldab = ABf.shape
    nrhs, ldb = B.shape
    ABd = torch.from_numpy(np.ascontiguousarray(ABf)).to(DEV)
    ipd = torch.from_numpy(np.ascontiguousarray(ipiv, dtype=np.int32)).to(DEV)
    Bd = torch.from_numpy(np.ascontiguousarray(B)).to(DEV)
    rc = bandlu.gbtrs(n, kl, ku, nrhs, ABd, ldab, ipd, Bd, ldb)
    torch.cuda.synchronize()
    assert rc == 0, rc
    return Bd.cpu().numpy()


def assert_same_solution(got, ref):
    nan_g, nan_r = np.isnan(got), np.isnan(ref)
    assert np.array_equal(nan_g, nan_r)
    if not np.array_equal(got[~nan_g].view(np.int64), ref[~nan_r].view(np.int64)):
        d = np.argwhere(got.view(np.int64) != ref.view(np.int64))[0]
        raise AssertionError(f"solution not bit-identical first at {tuple(d)}: {got[tuple(d)]!r} vs {ref[tuple(d)]!r}")


# one-warp windows of 1, 2 and 4 registers per lane (kl+ku+1 <= 128); above, the CTA-wide window:
# 256 threads with one register (kw+33 <= 256), 512 threads with one or two, n below and far above
# the window (the refills), a sweep of each size in one solve; kl+ku > 991: the shared-memory ring
@pytest.mark.parametrize("n,kl,ku,nrhs", [(1, 0, 0, 1), (2, 1, 0, 1), (17, 3, 5, 3), (300, 2, 2, 1), (512, 3, 3, 2),
                                          (1000, 16, 16, 5), (700, 0, 12, 1), (700, 12, 0, 1), (600, 40, 40, 2),
                                          (500, 60, 60, 1), (100, 60, 80, 1), (900, 64, 100, 2), (1300, 90, 120, 1),
                                          (400, 100, 150, 1), (350, 200, 250, 1),
                                          (250, 300, 300, 1), (3000, 300, 300, 2), (2100, 7, 600, 1),
                                          (1500, 100, 900, 1)])
def test_gbtrs_matches_oracle(n, kl, ku, nrhs):
    A = banded(n, kl, ku, seed=3 * n + kl + ku, dist="normal").numpy()
    ABf, ipiv, info, _ = oracle.gbtrf(oracle.dense_to_band(A, kl, ku), kl, ku)
    B = np.random.default_rng(n + nrhs).standard_normal((nrhs, n + 3))   # ldb = n + 3
    B[:, :2] = 0.0                                                       # the zero skips
    ref = oracle.gbtrs(ABf, ipiv, kl, ku, B)
    assert_same_solution(gbtrs_gpu(ABf, ipiv, kl, ku, B), ref)


@pytest.mark.parametrize("n,kl,ku", [(400, 5, 4), (600, 70, 90), (700, 200, 250)])
def test_gbtrs_zero_right_hand_sides_and_singular_factor(n, kl, ku):
    A = banded(n, kl, ku, seed=77).numpy()
    ABf, ipiv, info, _ = oracle.gbtrf(oracle.dense_to_band(A, kl, ku), kl, ku)
    B = np.zeros((3, n))
    B[1, 7] = 1.0
    assert_same_solution(gbtrs_gpu(ABf, ipiv, kl, ku, B), oracle.gbtrs(ABf, ipiv, kl, ku, B))
    A[:, 100] = 0.0                                                      # singular: infinities, NaNs
    ABf, ipiv, info, _ = oracle.gbtrf(oracle.dense_to_band(A, kl, ku), kl, ku)
    assert info > 0
    B = np.random.default_rng(2).standard_normal((1, n))
    assert_same_solution(gbtrs_gpu(ABf, ipiv, kl, ku, B), oracle.gbtrs(ABf, ipiv, kl, ku, B))


def run_solve(A, B, ldab):
    n, lda = A.shape
    nrhs, ldb = B.shape
    Ad, Bd = A.to(DEV), torch.from_numpy(np.ascontiguousarray(B)).to(DEV)
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=DEV)
    ipiv = torch.zeros(max(n, 1), dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, kl, ku = bandlu.dispatch_solve(Ad, n, lda, Bd, ldb, nrhs, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    return rc, kl, ku, Bd.cpu().numpy(), int(info.item())


@pytest.mark.parametrize("n,kl,ku", [(512, 3, 3), (4096, 16, 16), (1500, 40, 20)])
def test_dispatch_solve_matches_oracle(n, kl, ku):
    A = banded(n, kl, ku, seed=n + 1)
    ldab = 2 * kl + ku + 1
    B = np.random.default_rng(n).uniform(-1, 1, (2, n))
    rc, gkl, gku, X, info = run_solve(A, B, ldab)
    r = oracle.dispatch_lu(A.numpy(), ldab)
    assert (rc, gkl, gku, info) == (r["status"], r["kl"], r["ku"], r["info"]) == (0, kl, ku, 0)
    ref = oracle.gbtrs(r["AB"], r["ipiv"], kl, ku, B)
    assert_same_solution(X, ref)
    An = A.numpy()
    r = np.max(np.abs(An @ X[0] - B[0]))
    assert r / (np.max(np.sum(np.abs(An), axis=1)) * np.max(np.abs(X[0])) * n * 2.0 ** -53) <= 10.0


def test_dispatch_solve_declines_and_skips_singular():
    n = 300
    A = banded(n, 2, 3, seed=4)
    A[n - 1, 0] = 1e-3                                                   # not banded: B untouched
    B = np.random.default_rng(0).standard_normal((1, n))
    rc, kl, ku, X, info = run_solve(A, B, 8)
    assert rc == bandlu.BANDLU_NOT_BANDED and np.array_equal(X, B) and info == -5
    A = banded(n, 2, 3, seed=4)
    A[:, 50] = 0.0                                                       # singular: B untouched, info > 0
    rc, kl, ku, X, info = run_solve(A, B, 8)
    assert rc == 0 and info == 51 and np.array_equal(X, B)


# --------------------------------------------------------------------------------------------
# dispatch_lu and dispatch_lu_batched
# --------------------------------------------------------------------------------------------

def run_dispatch(A: torch.Tensor, ldab: int):
    n, lda = A.shape
    Ad = A.to(DEV)
    AB = torch.full((n, ldab), -3.0, dtype=torch.float64, device=DEV)
    ipiv = torch.full((max(n, 1),), -1, dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, kl, ku = bandlu.dispatch_lu(Ad, n, lda, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    return rc, kl, ku, AB.cpu().numpy(), ipiv.cpu().numpy()[:n], int(info.item())


@pytest.mark.parametrize("n,kl,ku,ldab", [(512, 3, 3, 10), (600, 2, 9, 20), (300, 20, 20, 61), (100, 0, 0, 1)])
def test_dispatch_lu_matches_oracle(n, kl, ku, ldab):
    A = banded(n, kl, ku, seed=n + ldab)
    rc, gkl, gku, AB, ipiv, info = run_dispatch(A, ldab)
    r = oracle.dispatch_lu(A.numpy(), ldab)
    assert (rc, gkl, gku) == (r["status"], r["kl"], r["ku"]) == (0, kl, ku)
    assert_factor_parity(AB, ipiv, info, r["AB"], r["ipiv"], r["info"])


def test_dispatch_lu_declines_stray_entry_and_leaves_outputs():
    n = 400
    A = banded(n, 2, 3, seed=4)
    A[n - 1, 0] = 1e-3
    rc, kl, ku, AB, ipiv, info = run_dispatch(A, 8)
    assert (rc, kl, ku) == (bandlu.BANDLU_NOT_BANDED, n - 1, 3)
    assert np.all(AB == -3.0) and np.all(ipiv == -1) and info == -5


def test_dispatch_lu_declines_when_storage_too_small():
    A = banded(300, 4, 4, seed=1)
    rc, kl, ku, *_ = run_dispatch(A, 12)            # needs 13
    assert (rc, kl, ku) == (bandlu.BANDLU_NOT_BANDED, 4, 4)


def run_batched(A: torch.Tensor, ldab: int):
    batch, n, lda = A.shape
    Ad = A.to(DEV)
    AB = torch.full((batch, n, ldab), -3.0, dtype=torch.float64, device=DEV)
    ipiv = torch.full((batch, n), -1, dtype=torch.int32, device=DEV)
    kl = torch.full((batch,), -1, dtype=torch.int32, device=DEV)
    ku = torch.full((batch,), -1, dtype=torch.int32, device=DEV)
    info = torch.full((batch,), -1, dtype=torch.int32, device=DEV)
    status = torch.full((batch,), -1, dtype=torch.int32, device=DEV)
    rc = bandlu.dispatch_lu_batched(Ad, n, lda, n * lda, batch, AB, ldab, n * ldab, ipiv, n, kl, ku, info, status)
    torch.cuda.synchronize()
    assert rc == 0
    return dict(AB=AB.cpu().numpy(), ipiv=ipiv.cpu().numpy(), kl=kl.cpu().numpy(), ku=ku.cpu().numpy(),
                info=info.cpu().numpy(), status=status.cpu().numpy())


def compare_batched(got, ref):
    for key in ("kl", "ku", "status", "info"):
        assert np.array_equal(got[key], ref[key]), key
    banded_idx = np.nonzero(ref["status"] == 0)[0]
    for b in banded_idx:
        assert_factor_parity(got["AB"][b], got["ipiv"][b], int(got["info"][b]), ref["AB"][b], ref["ipiv"][b],
                             int(ref["info"][b]))
    for b in np.nonzero(ref["status"] != 0)[0]:
        assert np.all(got["AB"][b] == -3.0) and np.all(got["ipiv"][b] == -1)


def test_batched_mixed_matrices():
    n, ldab = 64, 12
    mats = [banded(n, 2, 2, seed=s, boost=4.0) for s in range(5)]
    mats.append(banded(n, 3, 5, seed=7))            # uses the whole storage
    mats.append(banded(n, 4, 4, seed=8))            # needs 13 > 12: declined
    s = banded(n, 1, 1, seed=9); s[n - 1, 0] = 2.0
    mats.append(s)                                   # stray entry: declined
    z = torch.zeros((n, n), dtype=torch.float64)
    mats.append(z)                                   # all zero: kl = ku = 0, zero pivots
    d = banded(n, 0, 0, seed=10); d[5, 5] = 0.0
    mats.append(d)                                   # diagonal with a zero pivot
    A = torch.stack(mats)
    got = run_batched(A, ldab)
    ref = oracle.dispatch_lu_batched(A.numpy(), ldab)
    compare_batched(got, ref)
    assert list(got["status"][6:8]) == [1, 1]


def test_batched_many_small_varied_bands():
    # more matrices than the persistent kernel has hand-off slots, bands from diagonal
    # to wider than a register window, storage taller than the band (zeroed rows)
    rng = np.random.default_rng(3)
    n, ldab, batch = 40, 16, 2500
    mats = []
    for b in range(batch):
        kl, ku = int(rng.integers(0, 5)), int(rng.integers(0, 6))
        mats.append(banded(n, kl, ku, seed=b, boost=3.0 * float(rng.integers(0, 2))))
    A = torch.stack(mats)
    got = run_batched(A, ldab)
    ref = oracle.dispatch_lu_batched(A.numpy(), ldab)
    compare_batched(got, ref)


@pytest.mark.parametrize("batch,n,kl,ku,lda", [(37, 256, 2, 2, 256), (16, 100, 3, 1, 101), (8, 1, 0, 0, 1),
                                               (5, 700, 10, 10, 700),
                                               # column windows: kl = 7 in 8 row registers (ldab 16),
                                               # and 8 matrices per warp (ldab 3)
                                               (12, 50, 7, 1, 50), (33, 64, 1, 0, 64)])
def test_batched_matches_oracle(batch, n, kl, ku, lda):
    A = make_dense(n, kl, ku, dist="uniform", diag_boost=0.0, seed=batch + n, batch=batch, lda=lda)
    ldab = 2 * kl + ku + 1
    got = run_batched(A, ldab)
    ref = oracle.dispatch_lu_batched(A.numpy(), ldab)
    compare_batched(got, ref)
