"""Pins for the CPU oracle against facts fixed outside the oracle itself.

Each group checks one oracle function against something other than its own
formula: special cases, an independent characterisation, a library routine
(numpy / scipy / LAPACK), exact rational arithmetic, a closed form, or values
the paper prints.  A plausible slip in the oracle (a dropped term, a wrong
sign, a transposed index, an off-by-one in the band bookkeeping) fails at
least one of them.
"""
import itertools
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import scipy.linalg
import scipy.linalg.lapack as lapack

from paper_2608_22099_gb300.workloads import make_dense

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_banded(n, kl, ku, seed, boost=0.0, dist="uniform", lda=None):
    return make_dense(n, kl, ku, dist=dist, diag_boost=boost, seed=seed, lda=lda).numpy()


# ----------------------------------------------------------------------------------------------
# Detection (Sec. III-A Eq. IC-N2; element inspection as in Listing 1 / Listing 2)
# ----------------------------------------------------------------------------------------------

def bandwidth_by_tril_triu(A):
    """Independent characterisation: kl is the least k >= 0 with tril(A, -(k+1)) == 0,
    ku the least k >= 0 with triu(A, k+1) == 0 (the istril/istriu tests of Listing 1)."""
    n = A.shape[0]
    kl = next(k for k in range(n + 1) if not np.any(np.tril(A, -(k + 1)) != 0))
    ku = next(k for k in range(n + 1) if not np.any(np.triu(A, k + 1) != 0))
    return kl, ku


@pytest.mark.parametrize("n", [1, 2, 3, 7, 33])
def test_detect_special_cases(oracle_mod, n):
    z = np.zeros((n, n))
    assert oracle_mod.detect_bandwidth(z) == (0, 0)
    full = np.random.default_rng(n).uniform(0.5, 1.0, (n, n))
    assert oracle_mod.detect_bandwidth(full) == (n - 1, n - 1)
    assert oracle_mod.detect_bandwidth(np.diag(np.arange(1.0, n + 1))) == (0, 0)
    s = z.copy(); s[n - 1, 0] = 1e-3
    assert oracle_mod.detect_bandwidth(s) == (n - 1, 0)
    s = z.copy(); s[0, n - 1] = -7.0
    assert oracle_mod.detect_bandwidth(s) == (0, n - 1)


def test_detect_empty(oracle_mod):
    assert oracle_mod.detect_bandwidth(np.zeros((0, 1))) == (0, 0)


def test_detect_ieee_zero_policy(oracle_mod):
    n = 6
    A = np.zeros((n, n))
    A[5, 0] = -0.0            # negative zero is zero
    assert oracle_mod.detect_bandwidth(A) == (0, 0)
    for v, pos, expect in [(np.nan, (4, 1), (3, 0)), (np.inf, (0, 3), (0, 3)), (-np.inf, (2, 0), (2, 0)),
                           (5e-324, (5, 2), (3, 0)), (-5e-324, (1, 5), (0, 4))]:
        B = A.copy(); B[pos] = v
        assert oracle_mod.detect_bandwidth(B) == expect, v


def test_detect_matches_tril_triu_random_patterns(oracle_mod):
    rng = np.random.default_rng(5)
    for trial in range(400):
        n = int(rng.integers(1, 24))
        A = np.where(rng.random((n, n)) < rng.uniform(0.0, 0.3), rng.standard_normal((n, n)), 0.0)
        assert oracle_mod.detect_bandwidth(A) == bandwidth_by_tril_triu(A), trial


def test_detect_ignores_lda_padding(oracle_mod):
    n, lda = 9, 13
    A = rand_banded(n, 1, 2, seed=3, lda=lda)
    A[:, n:] = 1.0            # padding columns are not part of the matrix
    assert oracle_mod.detect_bandwidth(A) == (1, 2)


@pytest.mark.parametrize("n,kl,ku", [(512, 3, 3), (300, 16, 16), (257, 8, 64), (256, 2, 2), (100, 0, 5), (100, 5, 0)])
def test_detect_generator_invariant(oracle_mod, n, kl, ku):
    # the generator fills every diagonal -kl..ku with nonzeros (probability 1)
    A = rand_banded(n, kl, ku, seed=n + kl)
    assert oracle_mod.detect_bandwidth(A) == (kl, ku)


# ----------------------------------------------------------------------------------------------
# Conversion (Sec. III-A Eq. IC-N2; BandedMatrix(A) in Listing 2; LAPACK band storage)
# ----------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,kl,ku", [(1, 0, 0), (5, 1, 1), (17, 3, 8), (40, 0, 7), (40, 7, 0), (64, 16, 16)])
def test_band_round_trip(oracle_mod, n, kl, ku):
    A = rand_banded(n, kl, ku, seed=11)
    for ekl, eku in [(kl, ku), (kl + 2, ku + 1)]:      # any storage at least as wide as the band
        AB = oracle_mod.dense_to_band(A, ekl, eku)
        B = oracle_mod.band_to_dense(AB, ekl, eku)
        assert np.array_equal(A.view(np.int64), B.view(np.int64))


def test_band_layout_consumed_by_library_solver(oracle_mod):
    """scipy.linalg.solve_banded reads (l+u+1, n) storage with ab[u+i-j, j] = a[i, j]: rows
    kl..2kl+ku of the LAPACK layout.  Solving with it must reproduce the dense solve."""
    rng = np.random.default_rng(2)
    for n, kl, ku in [(30, 2, 5), (50, 7, 1), (64, 16, 16), (12, 0, 3)]:
        A = rand_banded(n, kl, ku, seed=n, boost=3.0)
        AB = oracle_mod.dense_to_band(A, kl, ku)            # shape (n, ldab): AB[j, r]
        ab = AB.T[kl:, :]                                   # (kl+ku+1, n)
        b = rng.standard_normal(n)
        x = scipy.linalg.solve_banded((kl, ku), ab, b)
        np.testing.assert_allclose(x, np.linalg.solve(A, b), rtol=1e-10, atol=1e-12)


def test_band_fill_and_corners_are_positive_zero(oracle_mod):
    n, kl, ku = 10, 3, 2
    A = rand_banded(n, kl, ku, seed=4)
    ldab = 2 * kl + ku + 1 + 2                               # extra rows are zeroed too
    AB = oracle_mod.dense_to_band(A, kl, ku, ldab)
    kv = kl + ku
    for j in range(n):
        for r in range(ldab):
            i = j - kv + r
            inside = kl <= r <= kv + kl and 0 <= i < n
            if not inside:
                assert AB[j, r] == 0.0 and not math.copysign(1.0, AB[j, r]) < 0, (j, r)
            else:
                assert AB[j, r] == A[i, j]


# ----------------------------------------------------------------------------------------------
# Banded LU (Sec. III-A Eq. S-N-N3; DGBTRF in Listing 2)
# ----------------------------------------------------------------------------------------------

def lapack_layout(AB):
    """(n, ldab) row-per-band-column array -> Fortran (ldab, n) array."""
    return np.asfortranarray(AB.T)


def test_gbtrf_matches_lapack_dgbtrf(oracle_mod):
    """LAPACK's dgbtrf on the same storage: same pivots and info, factors to rounding."""
    cases = [(1, 0, 0), (2, 1, 0), (8, 1, 1), (37, 3, 2), (64, 16, 16), (200, 8, 30), (300, 2, 2),
             (128, 0, 4), (128, 5, 0), (96, 31, 31), (150, 12, 3), (200, 40, 20)]
    for idx, (n, kl, ku) in enumerate(cases):
        for dist in ("uniform", "normal"):
            A = rand_banded(n, kl, ku, seed=100 + idx, dist=dist)
            AB = oracle_mod.dense_to_band(A, kl, ku)
            ABf, ipiv, info, _ = oracle_mod.gbtrf(AB, kl, ku)
            lu, piv, linfo = lapack.dgbtrf(lapack_layout(AB), kl, ku)
            assert linfo == info
            assert np.array_equal(ipiv, piv.astype(np.int32) + 1), (n, kl, ku, dist)
            ref = np.asarray(lu).T
            scale = np.max(np.abs(ref)) or 1.0
            assert np.max(np.abs(ABf - ref)) / scale < 1e-13, (n, kl, ku, dist)


# ----------------------------------------------------------------------------------------------
# The solve after the factorisation (the backslash of Listing 1; LAPACK xGBTRS)
# ----------------------------------------------------------------------------------------------

def test_gbtrs_matches_lapack_dgbtrs(oracle_mod):
    """LAPACK's dgbtrs on the same factors and right-hand sides: the same solution to rounding."""
    cases = [(1, 0, 0), (2, 1, 0), (8, 1, 1), (37, 3, 2), (64, 16, 16), (200, 8, 30), (128, 0, 4),
             (128, 5, 0), (96, 31, 31)]
    for idx, (n, kl, ku) in enumerate(cases):
        A = rand_banded(n, kl, ku, seed=300 + idx, dist="normal", boost=2.0)
        ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
        assert info == 0
        B = np.random.default_rng(idx).standard_normal((3, n))
        X = oracle_mod.gbtrs(ABf, ipiv, kl, ku, B)
        xl, linfo = lapack.dgbtrs(lapack_layout(ABf), kl, ku, B.T.copy(), ipiv - 1)
        assert linfo == 0
        assert np.max(np.abs(X - xl.T)) <= 1e-12 * max(np.max(np.abs(xl)), 1.0), (n, kl, ku)


def test_gbtrs_backward_error(oracle_mod):
    """||A X - B|| / (||A|| ||X|| n eps) stays small, against a library dense product."""
    for idx, (n, kl, ku) in enumerate([(300, 4, 6), (500, 16, 16), (400, 40, 3)]):
        A = rand_banded(n, kl, ku, seed=400 + idx, dist="uniform")
        ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
        B = np.random.default_rng(idx).uniform(-1, 1, (2, n))
        X = oracle_mod.gbtrs(ABf, ipiv, kl, ku, B)
        for c in range(2):
            r = np.max(np.abs(A @ X[c] - B[c]))
            bound = np.max(np.sum(np.abs(A), axis=1)) * np.max(np.abs(X[c])) * n * 2.0 ** -53
            assert r / bound <= 10.0, (n, kl, ku, r / bound)


def test_gbtrs_exact_rational_solutions(oracle_mod):
    """Small integer systems solved exactly in rationals: the oracle's solution to rounding."""
    from fractions import Fraction
    rng = np.random.default_rng(5)
    for trial in range(40):
        n, kl, ku = int(rng.integers(1, 9)), int(rng.integers(0, 3)), int(rng.integers(0, 3))
        A = np.zeros((n, n))
        for i in range(n):
            for j in range(max(0, i - kl), min(n, i + ku + 1)):
                A[i, j] = float(rng.integers(-4, 5))
            A[i, i] = float(rng.integers(5, 9)) * (1 if rng.random() < 0.5 else -1)
        b = rng.integers(-9, 10, n).astype(float)
        # exact elimination with rationals
        M = [[Fraction(int(A[i, j])) for j in range(n)] + [Fraction(int(b[i]))] for i in range(n)]
        for j in range(n):
            p = max(range(j, n), key=lambda r: abs(M[r][j]))
            M[j], M[p] = M[p], M[j]
            for r in range(j + 1, n):
                f = M[r][j] / M[j][j]
                M[r] = [x - f * y for x, y in zip(M[r], M[j])]
        x = [Fraction(0)] * n
        for j in reversed(range(n)):
            x[j] = (M[j][n] - sum(M[j][k] * x[k] for k in range(j + 1, n))) / M[j][j]
        ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
        X = oracle_mod.gbtrs(ABf, ipiv, kl, ku, b[None])[0]
        ex = np.array([float(v) for v in x])
        assert np.max(np.abs(X - ex)) <= 1e-13 * max(np.max(np.abs(ex)), 1.0), (trial, n, kl, ku)


@pytest.mark.parametrize("n", [1, 2, 10, 100])
def test_gbtrs_tridiagonal_closed_form(oracle_mod, n):
    """tridiag(-1, 2, -1) x = e_1 has x_i = (n - i) / (n + 1) (0-based i)."""
    A = np.diag(np.full(n, 2.0)) - np.diag(np.ones(n - 1), 1) - np.diag(np.ones(n - 1), -1)
    ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, 1, 1), 1, 1)
    e1 = np.zeros(n); e1[0] = 1.0
    X = oracle_mod.gbtrs(ABf, ipiv, 1, 1, e1[None])[0]
    ex = (n - np.arange(n)) / (n + 1.0)
    assert np.max(np.abs(X - ex)) <= 4 * n * 2.0 ** -52


def test_gbtrs_zero_right_hand_side_and_layout(oracle_mod):
    n, kl, ku = 60, 3, 2
    A = rand_banded(n, kl, ku, seed=9, boost=1.0)
    ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
    Z = oracle_mod.gbtrs(ABf, ipiv, kl, ku, np.zeros((2, n)))
    assert np.all(Z == 0.0) and not np.any(np.signbit(Z))   # every step skipped: +0.0 stays +0.0
    B = np.random.default_rng(1).standard_normal((2, n + 5))  # ldb = n + 5: the padding is untouched
    X = oracle_mod.gbtrs(ABf, ipiv, kl, ku, B)
    assert np.array_equal(X[:, n:], B[:, n:])
    assert np.allclose(A @ X[0, :n], B[0, :n], atol=1e-12)


def factors_from_band(ABf, kl, ku):
    """U (dense, upper) and the multiplier matrix (dense, strictly lower) from band storage."""
    n = ABf.shape[0]
    kv = kl + ku
    U = np.zeros((n, n)); L = np.zeros((n, n))
    for j in range(n):
        for i in range(max(0, j - kv), j + 1):
            U[i, j] = ABf[j, kv + i - j]
        for t in range(1, min(kl, n - 1 - j) + 1):
            L[j + t, j] = ABf[j, kv + t]
    return U, L


def test_gbtrf_equals_dense_lu_exhaustive_small_patterns(oracle_mod):
    """Every sparsity pattern of a 3x3 matrix (and a sample of 4x4 ones), random values: the band
    factorisation equals plain dense elimination bit for bit (skipped operations are x - l*0)."""
    rng = np.random.default_rng(7)
    pats = [(n, bits) for n in (1, 2, 3) for bits in range(1 << (n * n))]
    pats += [(4, int(b)) for b in rng.integers(0, 1 << 16, 3000)]
    for n, bits in pats:
        mask = np.array([(bits >> k) & 1 for k in range(n * n)], dtype=bool).reshape(n, n)
        A = np.where(mask, rng.uniform(-1, 1, (n, n)), 0.0)
        check_dense_equivalence(oracle_mod, A)


def check_dense_equivalence(oracle_mod, A):
    kl, ku = oracle_mod.detect_bandwidth(A)
    AB = oracle_mod.dense_to_band(A, kl, ku)
    ABf, ipiv, info, _ = oracle_mod.gbtrf(AB, kl, ku)
    D, dpiv, dinfo = oracle_mod.getrf_dense(A)
    assert np.array_equal(ipiv, dpiv) and info == dinfo
    U, L = factors_from_band(ABf, kl, ku)
    assert np.array_equal(np.triu(D), U)
    assert np.array_equal(np.tril(D, -1), L)


def test_gbtrf_equals_dense_lu_random(oracle_mod):
    rng = np.random.default_rng(8)
    for trial in range(150):
        n = int(rng.integers(1, 65))
        kl = int(rng.integers(0, min(n, 12)))
        ku = int(rng.integers(0, min(n, 12)))
        A = rand_banded(n, kl, ku, seed=trial, dist="normal" if trial % 2 else "uniform")
        # knock out random entries (zero pivots, zero u's, uneven structure)
        A[rng.random((n, n)) < 0.15] = 0.0
        check_dense_equivalence(oracle_mod, A)


def dense_lu_to_getrf_form(D, piv):
    """Our dense LU keeps each multiplier column where it was computed; LAPACK's dgetrf applies
    the later interchanges to the earlier multiplier columns as well.  Convert for comparison."""
    D = D.copy()
    n = D.shape[0]
    for k in range(n):
        p = piv[k] - 1
        if p != k:
            D[[k, p], :k] = D[[p, k], :k]
    return D


def test_dense_lu_matches_lapack_dgetrf(oracle_mod):
    rng = np.random.default_rng(9)
    for n in (1, 2, 5, 16, 40, 90):
        A = rng.standard_normal((n, n))
        D, piv, info = oracle_mod.getrf_dense(A)
        lu, lpiv, linfo = lapack.dgetrf(A)
        assert info == linfo
        assert np.array_equal(piv, lpiv.astype(np.int32) + 1)
        np.testing.assert_allclose(dense_lu_to_getrf_form(D, piv), lu, rtol=1e-11, atol=1e-13)


def exact_lu(A):
    """Partial-pivoting elimination in exact rational arithmetic (first maximal |.| as pivot)."""
    n = len(A)
    M = [[Fraction(x) for x in row] for row in A]
    piv = []
    for j in range(n):
        p = max(range(j, n), key=lambda i: (abs(M[i][j]), -i))
        piv.append(p)
        if M[p][j] == 0:
            continue
        M[j][j:], M[p][j:] = M[p][j:], M[j][j:]
        for i in range(j + 1, n):
            l = M[i][j] / M[j][j]
            M[i][j] = l
            for c in range(j + 1, n):
                M[i][c] -= l * M[j][c]
    return M, piv


def test_gbtrf_against_exact_rational_elimination(oracle_mod):
    rng = np.random.default_rng(10)
    compared = 0
    for trial in range(60):
        n = int(rng.integers(2, 9))
        kl = int(rng.integers(0, n)); ku = int(rng.integers(0, n))
        A = np.zeros((n, n))
        for i in range(n):
            for j in range(max(0, i - kl), min(n, i + ku + 1)):
                A[i, j] = float(rng.integers(-9, 10))
        M, epiv = exact_lu(A.tolist())
        kl2, ku2 = oracle_mod.detect_bandwidth(A)
        ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl2, ku2), kl2, ku2)
        U, L = factors_from_band(ABf, kl2, ku2)
        if not np.array_equal(ipiv - 1, np.array(epiv)):
            continue                                      # an exact tie broken the other way by rounding
        compared += 1
        for i in range(n):
            for j in range(n):
                exact = float(M[i][j])
                got = U[i, j] if i <= j else L[i, j]
                assert abs(got - exact) <= 1e-12 * max(1.0, abs(exact)), (trial, i, j)
    assert compared >= 40


@pytest.mark.parametrize("n", [1, 2, 3, 10, 1000, 100000])
def test_gbtrf_closed_form_tridiagonal(oracle_mod, n):
    """tridiag(-1, 2, -1): no interchanges, u_jj = (j+2)/(j+1), l_{j+1,j} = -(j+1)/(j+2),
    superdiagonal -1, det = n + 1."""
    AB = np.zeros((n, 4))                                 # kl = ku = 1, ldab = 4, kv = 2
    AB[:, 2] = 2.0
    AB[1:, 1] = -1.0                                      # U(j-1, j): row kv-1
    AB[:-1, 3] = -1.0                                     # L(j+1, j): row kv+1
    ABf, ipiv, info, _ = oracle_mod.gbtrf(AB, 1, 1)
    j = np.arange(n)
    assert info == 0 and np.array_equal(ipiv, (j + 1).astype(np.int32))
    # each elimination step adds at most a few rounding errors to the running pivot, which the
    # recurrence u_{j+1} = 2 - 1/u_j carries forward undamped: allow (j+1) * 4 ulp
    tol = 4 * 2.0 ** -52 * (j + 1)
    assert np.all(np.abs(ABf[:, 2] - (j + 2) / (j + 1)) <= tol * (j + 2) / (j + 1))
    assert np.all(np.abs(ABf[:-1, 3] + (j[:-1] + 1) / (j[:-1] + 2)) <= tol[:-1])
    assert np.all(ABf[1:, 1] == -1.0) and np.all(ABf[:, 0] == 0.0)
    logdet = np.sum(np.log(ABf[:, 2]))
    assert abs(logdet - math.log(n + 1)) < 1e-13 * max(1, n) + 1e-14


def test_gbtrf_upper_triangular_and_diagonal(oracle_mod):
    for n, ku in [(20, 0), (20, 4), (64, 63)]:
        A = np.triu(rand_banded(n, 0, ku, seed=ku))
        AB = oracle_mod.dense_to_band(A, 0, ku)
        ABf, ipiv, info, _ = oracle_mod.gbtrf(AB, 0, ku)
        assert np.array_equal(ipiv, np.arange(1, n + 1, dtype=np.int32)) and info == 0
        assert np.array_equal(ABf, AB)                     # U = A, nothing else written


def test_gbtrf_forced_interchanges(oracle_mod):
    n = 12
    A = np.diag(np.full(n, 1e-3)) + np.diag(np.ones(n - 1), -1) + np.diag(np.full(n - 1, 0.5), 1)
    ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, 1, 1), 1, 1)
    assert info == 0
    assert np.array_equal(ipiv[:-1], np.arange(2, n + 1, dtype=np.int32))
    # the interchange pulls row j+1's superdiagonal into U's second superdiagonal (fill row)
    assert np.all(ABf[2:, 0] != 0.0)


def test_gbtrf_zero_pivot_sets_info_and_continues(oracle_mod):
    n, kl, ku = 9, 2, 1
    A = rand_banded(n, kl, ku, seed=21, boost=3.0)
    A[:, 4] = 0.0                                          # exact zero column 4
    ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
    assert info == 5 and ipiv[4] == 5
    check_dense_equivalence(oracle_mod, A)                 # and the later columns are still factored
    B = A.copy(); B[:, 2] = 0.0
    _, _, info2, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(B, kl, ku), kl, ku)
    assert info2 == 3                                      # the first zero pivot is reported


def test_gbtrf_pivot_comparison_order_with_nan(oracle_mod):
    # The pivot is the first candidate of largest modulus in the comparison order
    # of the running maximum (LAPACK's IDAMAX rule): a later candidate replaces the
    # running best only if strictly larger, which a NaN never is.
    n, kl, ku = 3, 2, 1
    def piv(col0):
        A = np.eye(n) * 3.0
        A[:, 0] = col0
        A[0, 1] = 0.5
        ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
        return int(ipiv[0]), info
    assert piv([1.0, np.nan, 2.0]) == (3, 0)          # NaN skipped, 2 > 1 taken
    assert piv([np.nan, 5.0, -7.0]) == (1, 0)         # a NaN first candidate is kept
    assert piv([0.0, np.nan, 0.0]) == (1, 1)          # NaN never beats zero: zero pivot
    assert piv([-0.0, 0.0, np.inf])[0] == 3           # signed zeros tie, infinity wins


def test_gbtrf_invariants_and_backward_error(oracle_mod):
    rng = np.random.default_rng(12)
    for trial in range(40):
        n = int(rng.integers(1, 300)); kl = int(rng.integers(0, 20)); ku = int(rng.integers(0, 20))
        A = rand_banded(n, kl, ku, seed=500 + trial, dist="normal")
        AB = oracle_mod.dense_to_band(A, kl, ku)
        ABf, ipiv, info, flops = oracle_mod.gbtrf(AB, kl, ku)
        kv = kl + ku
        for j in range(n):
            km = min(kl, n - 1 - j)
            assert j + 1 <= ipiv[j] <= j + 1 + km
            assert np.all(np.abs(ABf[j, kv + 1: kv + 1 + km]) <= 1.0)
            assert np.all(ABf[j, kv + 1 + km:] == 0.0)      # below the matrix: untouched zeros
        assert 0 <= flops <= sum(1 + min(kl, n - 1 - j) * (1 + 2 * min(kv, n - 1 - j)) for j in range(n))
        assert oracle_mod.backward_error(A, ABf, ipiv, kl, ku) <= 10.0, trial


def test_band_residual_matches_dense_reconstruction(oracle_mod):
    rng = np.random.default_rng(13)
    for n, kl, ku in [(30, 3, 2), (45, 6, 6), (20, 0, 3), (25, 4, 0)]:
        A = rand_banded(n, kl, ku, seed=n)
        ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
        U, L = factors_from_band(ABf, kl, ku)
        M = U.copy()
        for j in range(n - 1, -1, -1):                    # A = P0 L0 P1 L1 ... U, rebuilt with matmul
            Lj = np.eye(n); Lj[:, j] += L[:, j]
            M = Lj @ M
            p = ipiv[j] - 1
            M[[j, p]] = M[[p, j]]
        dense_res = np.max(np.sum(np.abs(A - M), axis=1))
        r, an = oracle_mod.band_residual(A, ABf, ipiv, kl, ku)
        assert an == np.max(np.sum(np.abs(A), axis=1))
        assert abs(r - dense_res) <= 1e-12 * an
        # a wrong multiplier must show up in the residual
        bad = ABf.copy(); bad[n // 2, kl + ku + 1 if kl else kl + ku] += 1e-6
        r_bad, _ = oracle_mod.band_residual(A, bad, ipiv, kl, ku)
        assert r_bad > 1e-7


def test_flop_count_closed_form_without_interchanges(oracle_mod):
    n, kl, ku = 512, 3, 3
    A = rand_banded(n, kl, ku, seed=1001, boost=12.0)
    _, ipiv, info, flops = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, kl, ku), kl, ku)
    assert np.array_equal(ipiv, np.arange(1, n + 1, dtype=np.int32))
    expect = sum(1 + min(kl, n - 1 - j) + 2 * min(kl, n - 1 - j) * min(ku, n - 1 - j) for j in range(n))
    assert flops == expect


# ----------------------------------------------------------------------------------------------
# Dispatch predicate (Eq. su-con) and the whole strategy (Sec. II-A, Listing 2)
# ----------------------------------------------------------------------------------------------

def test_predicate_worked_cases(oracle_mod):
    # every banded workload shape is worth specialising; the stray-entry control is not
    for n, kl, ku in [(512, 3, 3), (4096, 16, 16), (16384, 8, 64), (256, 2, 2), (32768, 256, 256), (10000, 100, 100)]:
        assert oracle_mod.is_banded(n, kl, ku, 2 * kl + ku + 1)
        assert not oracle_mod.is_banded(n, kl, ku, 2 * kl + ku)          # storage too small
    assert not oracle_mod.is_banded(16384, 16383, 64, 10 ** 9)
    assert not oracle_mod.is_banded(1, 0, 0, 1) and not oracle_mod.is_banded(2, 0, 0, 1)
    assert oracle_mod.is_banded(3, 0, 0, 1)
    # dense n x n: never
    for n in (3, 10, 100, 1000):
        assert not oracle_mod.is_banded(n, n - 1, n - 1, 10 ** 9)


def _threshold_cases():
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "predicate_threshold_cases.txt")
    rows = []
    with open(path) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                kl, ku, n_min = (int(x) for x in line.split())
                rows.append((kl, ku, n_min))
    return rows


def test_predicate_hand_worked_thresholds(oracle_mod):
    """The smallest n that takes the band path, worked by hand from the operation counts of
    Eqs. IC-N2, S-N-N3 and D-N3 (tests/golden/predicate_threshold_cases.txt): n_min passes,
    n_min - 1 and every smaller n decline."""
    cases = _threshold_cases()
    assert len(cases) == 7
    for kl, ku, n_min in cases:
        ldab = 2 * kl + ku + 1
        assert oracle_mod.is_banded(n_min, kl, ku, ldab), (kl, ku, n_min)
        assert not oracle_mod.is_banded(n_min - 1, kl, ku, ldab), (kl, ku, n_min)
        assert not any(oracle_mod.is_banded(m, kl, ku, ldab) for m in range(max(1, n_min - 50), n_min - 1))


def test_predicate_against_exact_rational_cost_model(oracle_mod):
    rng = np.random.default_rng(14)
    for _ in range(2000):
        n = int(rng.integers(1, 5000)); kl = int(rng.integers(0, n)); ku = int(rng.integers(0, n))
        I = Fraction(n * n); C = Fraction(n * (kl + ku + 1)); f = Fraction(n * kl * (2 * (kl + ku) + 1))
        F = Fraction(2, 3) * n ** 3
        assert oracle_mod.is_banded(n, kl, ku, 2 * kl + ku + 1) == (I + C + f < F)


def test_dispatch_lu_single_and_batched(oracle_mod):
    A = rand_banded(64, 2, 3, seed=31)
    r = oracle_mod.dispatch_lu(A, ldab=8)
    assert r["status"] == 0 and (r["kl"], r["ku"]) == (2, 3)
    ABf, ipiv, info, _ = oracle_mod.gbtrf(oracle_mod.dense_to_band(A, 2, 3), 2, 3)
    assert np.array_equal(r["AB"], ABf) and np.array_equal(r["ipiv"], ipiv) and r["info"] == info
    A2 = A.copy(); A2[63, 0] = 1e-3
    r2 = oracle_mod.dispatch_lu(A2, ldab=8)
    assert r2["status"] == 1 and r2["kl"] == 63 and np.all(r2["AB"] == 0.0)
    Ab = np.stack([A, A2, rand_banded(64, 1, 1, seed=5)])
    rb = oracle_mod.dispatch_lu_batched(Ab, ldab=8)
    assert list(rb["status"]) == [0, 1, 0] and list(rb["kl"]) == [2, 63, 1]


# ----------------------------------------------------------------------------------------------
# Values the paper prints (Sec. IV-B)
# ----------------------------------------------------------------------------------------------

def read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                k, v = line.split("=")
                vals[k.strip()] = float(v)
    return vals


def test_paper_memory_figures(oracle_mod):
    g = read_golden("paper_memory_fig5_fig6.txt")
    n, kl, ku = int(g["n"]), int(g["kl"]), int(g["ku"])
    mib = 2.0 ** 20
    # dense LU: the n x n copy plus n 8-byte pivots
    assert round((8 * n * n + 8 * n) / mib, 2) == g["dense_lu_mib"]
    # structure-aware: three n x ldab band arrays plus the pivots; reproduces the printed figure
    # only with LAPACK's pivoting height ldab = 2*kl + ku + 1
    ldab = oracle_mod.ldab_for(kl, ku)
    assert round((3 * 8 * ldab * n + 8 * n) / mib, 2) == g["structured_lu_mib"]
    assert round((3 * 8 * (kl + ku + 1) * n + 8 * n) / mib, 2) != g["structured_lu_mib"]
    assert oracle_mod.is_banded(n, kl, ku, ldab)


def test_gbtrf_ignores_garbage_in_fill_rows(oracle_mod):
    n, kl, ku = 40, 4, 3
    A = rand_banded(n, kl, ku, seed=77)
    AB = oracle_mod.dense_to_band(A, kl, ku)
    ref = oracle_mod.gbtrf(AB, kl, ku)
    G = AB.copy(); G[:, :kl] = 123.0
    got = oracle_mod.gbtrf(G, kl, ku)
    assert np.array_equal(ref[0], got[0]) and np.array_equal(ref[1], got[1])


# ----------------------------------------------------------------------------------------------
# Triangular and diagonal branches of the backslash dispatch (Listing 1, Sec. I-A)
# ----------------------------------------------------------------------------------------------

def band_triangle(n, k, lower, seed, boost=2.0, dist="uniform"):
    """Row-major n x n triangle with bandwidth k (the other triangle zero)."""
    A = rand_banded(n, k if lower else 0, 0 if lower else k, seed=seed, dist=dist, boost=boost)
    return A


@pytest.mark.parametrize("lower", [True, False])
def test_tbsv_matches_library_triangular_solve(oracle_mod, lower):
    """LAPACK's dtrtrs (scipy solve_triangular) on the same triangle: the same solution to rounding."""
    for idx, (n, k) in enumerate([(1, 0), (2, 1), (9, 3), (64, 16), (150, 40), (120, 119)]):
        A = band_triangle(n, k, lower, seed=700 + idx, boost=3.0)
        B = np.random.default_rng(idx).standard_normal((3, n))
        X, info = oracle_mod.tbsv_dense(A, lower, k, B)
        assert info == 0
        ref = scipy.linalg.solve_triangular(A, B.T, lower=lower, check_finite=False).T
        assert np.max(np.abs(X - ref)) <= 1e-12 * max(np.max(np.abs(ref)), 1.0), (n, k, lower)


@pytest.mark.parametrize("lower", [True, False])
def test_tbsv_exact_rational_solutions(oracle_mod, lower):
    """Integer triangles with power-of-two diagonals and small integer right-hand sides: every
    intermediate value is an exact binary fraction, so the oracle must return the rational
    solution exactly."""
    rng = np.random.default_rng(11 if lower else 12)
    for trial in range(60):
        n, k = int(rng.integers(1, 10)), int(rng.integers(0, 4))
        A = np.zeros((n, n))
        for i in range(n):
            for j in range(n):
                if (lower and 0 < i - j <= k) or (not lower and 0 < j - i <= k):
                    A[i, j] = float(rng.integers(-3, 4))
            A[i, i] = float(2 ** int(rng.integers(0, 3))) * (1 if rng.random() < 0.5 else -1)
        b = rng.integers(-9, 10, n).astype(float)
        Af = [[Fraction(int(A[i, j])) for j in range(n)] for i in range(n)]
        x = [Fraction(int(v)) for v in b]
        order = range(n) if lower else range(n - 1, -1, -1)
        for j in order:  # textbook substitution in rationals
            x[j] = x[j] / Af[j][j]
            for i in range(n):
                if (lower and i > j) or (not lower and i < j):
                    x[i] -= Af[i][j] * x[j]
        assert all(float(v) == v for v in x)  # exactly representable
        X, info = oracle_mod.tbsv_dense(A, lower, k, b)
        assert info == 0
        assert [Fraction(v) for v in X[0]] == x, (trial, n, k)


def test_tbsv_bidiagonal_closed_form(oracle_mod):
    """Unit bidiagonal with -1 next to the diagonal: the solution is the running sum of b
    (prefix sums for the lower, suffix sums for the upper triangle), exact in integers."""
    n = 200
    b = np.random.default_rng(3).integers(-50, 51, n).astype(float)
    L = np.eye(n) - np.eye(n, k=-1)
    X, info = oracle_mod.tbsv_dense(L, True, 1, b)
    assert info == 0 and np.array_equal(X[0], np.cumsum(b))
    U = np.eye(n) - np.eye(n, k=1)
    X, info = oracle_mod.tbsv_dense(U, False, 1, b)
    assert info == 0 and np.array_equal(X[0], np.cumsum(b[::-1])[::-1])


@pytest.mark.parametrize("lower", [True, False])
def test_tbsv_zero_diagonal_sets_info_and_leaves_b(oracle_mod, lower):
    """xTRTRS: the first exact zero on the diagonal is reported (1-based) and B is untouched."""
    n, k = 30, 4
    A = band_triangle(n, k, lower, seed=5)
    A[17, 17] = 0.0
    A[23, 23] = -0.0
    B = np.random.default_rng(1).standard_normal((2, n))
    X, info = oracle_mod.tbsv_dense(A, lower, k, B)
    assert info == 18
    assert np.array_equal(X, B)


@pytest.mark.parametrize("lower", [True, False])
def test_tbsv_reads_only_its_band(oracle_mod, lower):
    """Entries outside the triangle's band (NaN here) are never read; an exact zero in b is
    neither divided nor used (a -0.0 stays -0.0)."""
    n, k = 40, 3
    A = band_triangle(n, k, lower, seed=9)
    G = A.copy()
    for i in range(n):
        for j in range(n):
            if (lower and not 0 <= i - j <= k) or (not lower and not 0 <= j - i <= k):
                G[i, j] = np.nan
    b = np.random.default_rng(2).standard_normal(n)
    X1, _ = oracle_mod.tbsv_dense(A, lower, k, b)
    X2, _ = oracle_mod.tbsv_dense(G, lower, k, b)
    assert np.array_equal(X1.view(np.int64), X2.view(np.int64))
    z = np.zeros(n)
    z[0 if not lower else n - 1] = -0.0
    X, _ = oracle_mod.tbsv_dense(A, lower, k, -z)
    assert np.array_equal(X.view(np.int64), (-z)[None].view(np.int64))


def test_diag_solve_is_the_ieee_quotient(oracle_mod):
    """Diagonal(A) \\ B divides each row by its diagonal entry: numpy's division bit for bit;
    a zero diagonal entry is reported and leaves B untouched."""
    rng = np.random.default_rng(4)
    n = 300
    d = rng.standard_normal(n) * np.exp(rng.uniform(-30, 30, n))
    A = np.diag(d)
    B = rng.standard_normal((4, n))
    X, info = oracle_mod.diag_solve(A, B)
    assert info == 0
    assert np.array_equal(X.view(np.int64), (B / d).view(np.int64))
    A[100, 100] = 0.0
    X, info = oracle_mod.diag_solve(A, B)
    assert info == 101 and np.array_equal(X, B)


def test_classify_follows_the_order_of_listing_1(oracle_mod):
    """istril and istriu: diagonal; istril: lower; istriu: upper; otherwise LU (band path when
    the dispatch predicate accepts, dense otherwise).  Worked cases of each branch."""
    K = oracle_mod
    assert K.classify(100, 0, 0, 1) == K.KIND_DIAGONAL
    assert K.classify(100, 5, 0, 1) == K.KIND_LOWER  # triangles need no band storage
    assert K.classify(100, 0, 7, 1) == K.KIND_UPPER
    assert K.classify(100, 99, 0, 1) == K.KIND_LOWER  # a full triangle too
    assert K.classify(100, 3, 2, 9) == K.KIND_BANDED
    assert K.classify(100, 3, 2, 8) == K.KIND_DENSE  # no room for the band
    assert K.classify(10, 8, 8, 100) == K.KIND_DENSE  # the predicate declines
    assert K.classify(1, 0, 0, 1) == K.KIND_DIAGONAL
    for kl, ku in itertools.product(range(4), range(4)):
        A = rand_banded(12, kl, ku, seed=kl * 4 + ku, boost=4.0)
        got = K.dispatch_backslash(A, np.ones(12), 2 * kl + ku + 1)
        assert got["kind"] == K.classify(12, kl, ku, 2 * kl + ku + 1)
        assert (got["kl"], got["ku"]) == (kl, ku)


def test_dispatch_backslash_runs_the_chosen_branch(oracle_mod):
    """Each kind's solution is that branch's own solve; the dense kind leaves B untouched."""
    K = oracle_mod
    rng = np.random.default_rng(8)
    n = 40
    B = rng.standard_normal((2, n))
    D = np.diag(rng.uniform(1, 2, n))
    r = K.dispatch_backslash(D, B, 1)
    assert r["kind"] == K.KIND_DIAGONAL and np.array_equal(r["X"], K.diag_solve(D, B)[0])
    L = band_triangle(n, 5, True, seed=1)
    r = K.dispatch_backslash(L, B, 1)
    assert r["kind"] == K.KIND_LOWER and np.array_equal(r["X"], K.tbsv_dense(L, True, 5, B)[0])
    U = band_triangle(n, 6, False, seed=2)
    r = K.dispatch_backslash(U, B, 1)
    assert r["kind"] == K.KIND_UPPER and np.array_equal(r["X"], K.tbsv_dense(U, False, 6, B)[0])
    A = rand_banded(n, 3, 4, seed=3)
    r = K.dispatch_backslash(A, B, 11)
    ABf, ipiv, info, _ = K.gbtrf(K.dense_to_band(A, 3, 4), 3, 4)
    assert r["kind"] == K.KIND_BANDED and r["info"] == info == 0
    assert np.array_equal(r["X"], K.gbtrs(ABf, ipiv, 3, 4, B))
    r = K.dispatch_backslash(A, B, 10)
    assert r["kind"] == K.KIND_DENSE and np.array_equal(r["X"], B)
    assert np.max(np.abs(A @ K.dispatch_backslash(A, B, 11)["X"][0] - B[0])) < 1e-10


# ----------------------------------------------------------------------------------------------
# Column-major input (the layout Listing 1 and Listing 2 operate on in Julia)
# ----------------------------------------------------------------------------------------------

@pytest.mark.parametrize("n,kl,ku,pad", [(1, 0, 0, 0), (2, 1, 0, 1), (9, 0, 4, 3), (40, 5, 2, 0), (64, 63, 1, 2),
                                         (100, 7, 30, 5)])
def test_column_major_detect_and_convert(oracle_mod, n, kl, ku, pad):
    """Column-major storage of M is the row-major array of M^T (padded rows): detection must give
    M's bandwidths by the tril/triu characterisation, and the conversion M's band storage as the
    row-major conversion produces it."""
    M = rand_banded(n, kl, ku, seed=n + kl + 5 * ku)
    Acm = np.zeros((n, n + pad))
    Acm[:, :n] = M.T
    Acm[:, n:] = np.nan  # padding is never read
    assert oracle_mod.detect_bandwidth_cm(Acm) == bandwidth_by_tril_triu(M) == (kl, ku)
    for ldab in (2 * kl + ku + 1, 2 * kl + ku + 4):
        AB = oracle_mod.dense_to_band_cm(Acm, kl, ku, ldab)
        assert np.array_equal(AB.view(np.int64), oracle_mod.dense_to_band(M, kl, ku, ldab).view(np.int64))
        assert np.array_equal(oracle_mod.band_to_dense(AB, kl, ku), M)
