"""The C-ABI library builds, loads and exports every entry point include/bandlu.h
declares; invalid arguments are rejected on the host before anything is
enqueued (no GPU needed: these calls never reach CUDA)."""
import ctypes
import os
import re

import pytest

from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300 import build as pbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER_DIR = os.path.join(ROOT, "include")


def declared_functions():
    names = []
    for h in sorted(os.listdir(HEADER_DIR)):
        if not h.endswith(".h"):
            continue
        text = open(os.path.join(HEADER_DIR, h)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?\w+\s*\*?\s*(\w+)\s*\(", text, flags=re.M):
            names.append(m.group(1))
    return names


def test_library_builds_and_exports_every_declared_symbol():
    path = pbuild.build()
    assert os.path.exists(path)
    lib = ctypes.CDLL(path)
    names = declared_functions()
    assert {"detect_bandwidth", "dense_to_band", "gbtrf", "gbtrs", "dispatch_lu", "dispatch_solve",
            "dispatch_lu_batched"} <= set(names)
    for name in names:
        assert hasattr(lib, name), name
    assert bandlu.version().startswith("bandlu")


DEV = 1 << 20  # a non-null placeholder address: never dereferenced by the host checks


@pytest.mark.parametrize("args,expect", [
    ((DEV, -1, 1, DEV, DEV), -2),
    ((0, 4, 4, DEV, DEV), -1),
    ((DEV, 4, 3, DEV, DEV), -3),
    ((DEV, 4, 4, 0, DEV), -4),
    ((DEV, 4, 4, DEV, 0), -5),
    ((DEV, 1 << 31, 1 << 31, DEV, DEV), -2),
])
def test_detect_bandwidth_argument_checks(args, expect):
    assert bandlu.detect_bandwidth(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, 1, 1, DEV, 4), -1),
    ((DEV, 3, 4, 1, 1, DEV, 4), -2),
    ((DEV, 4, -1, 1, 1, DEV, 4), -3),
    ((DEV, 4, 4, -1, 1, DEV, 4), -4),
    ((DEV, 4, 4, 1, -1, DEV, 4), -5),
    ((DEV, 4, 4, 1, 1, 0, 4), -6),
    ((DEV, 4, 4, 1, 1, DEV, 3), -7),
])
def test_dense_to_band_argument_checks(args, expect):
    assert bandlu.dense_to_band(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((-1, 1, 1, DEV, 4, DEV, DEV), -1),
    ((4, -1, 1, DEV, 4, DEV, DEV), -2),
    ((4, 1, -1, DEV, 4, DEV, DEV), -3),
    ((4, 1, 1, 0, 4, DEV, DEV), -4),
    ((4, 2, 1, DEV, 5, DEV, DEV), -5),
    ((4, 1, 1, DEV, 4, 0, DEV), -6),
    ((4, 1, 1, DEV, 4, DEV, 0), -7),
])
def test_gbtrf_argument_checks(args, expect):
    assert bandlu.gbtrf(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, DEV, 4, DEV, DEV), -1),
    ((DEV, -2, 4, DEV, 4, DEV, DEV), -2),
    ((DEV, 4, 2, DEV, 4, DEV, DEV), -3),
    ((DEV, 4, 4, 0, 4, DEV, DEV), -4),
    ((DEV, 4, 4, DEV, 0, DEV, DEV), -5),
    ((DEV, 4, 4, DEV, 4, 0, DEV), -6),
    ((DEV, 4, 4, DEV, 4, DEV, 0), -9),
])
def test_dispatch_lu_argument_checks(args, expect):
    rc, _, _ = bandlu.dispatch_lu(*args, stream=0)
    assert rc == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, 16, 2, DEV, 4, 16, DEV, 4, DEV, DEV, DEV, DEV), -1),
    ((DEV, 4, 4, 15, 2, DEV, 4, 16, DEV, 4, DEV, DEV, DEV, DEV), -4),
    ((DEV, 4, 4, 16, -1, DEV, 4, 16, DEV, 4, DEV, DEV, DEV, DEV), -5),
    ((DEV, 4, 4, 16, 2, DEV, 4, 15, DEV, 4, DEV, DEV, DEV, DEV), -8),
    ((DEV, 4, 4, 16, 2, DEV, 4, 16, DEV, 3, DEV, DEV, DEV, DEV), -10),
    ((DEV, 4, 4, 16, 2, DEV, 4, 16, DEV, 4, DEV, DEV, DEV, 0), -14),
])
def test_dispatch_lu_batched_argument_checks(args, expect):
    assert bandlu.dispatch_lu_batched(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((-1, 1, 1, 1, DEV, 4, DEV, DEV, 4), -1),
    ((4, -1, 1, 1, DEV, 4, DEV, DEV, 4), -2),
    ((4, 1, -1, 1, DEV, 4, DEV, DEV, 4), -3),
    ((4, 1, 1, -1, DEV, 4, DEV, DEV, 4), -4),
    ((4, 1, 1, 1, 0, 4, DEV, DEV, 4), -5),
    ((4, 2, 1, 1, DEV, 5, DEV, DEV, 4), -6),
    ((4, 1, 1, 1, DEV, 4, 0, DEV, 4), -7),
    ((4, 1, 1, 1, DEV, 4, DEV, 0, 4), -8),
    ((4, 1, 1, 1, DEV, 4, DEV, DEV, 3), -9),
])
def test_gbtrs_argument_checks(args, expect):
    assert bandlu.gbtrs(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, DEV, 4, 1, DEV, 4, DEV, DEV), -1),
    ((DEV, -2, 4, DEV, 4, 1, DEV, 4, DEV, DEV), -2),
    ((DEV, 4, 3, DEV, 4, 1, DEV, 4, DEV, DEV), -3),
    ((DEV, 4, 4, 0, 4, 1, DEV, 4, DEV, DEV), -4),
    ((DEV, 4, 4, DEV, 3, 1, DEV, 4, DEV, DEV), -5),
    ((DEV, 4, 4, DEV, 4, -1, DEV, 4, DEV, DEV), -6),
    ((DEV, 4, 4, DEV, 4, 1, 0, 4, DEV, DEV), -7),
    ((DEV, 4, 4, DEV, 4, 1, DEV, 0, DEV, DEV), -8),
    ((DEV, 4, 4, DEV, 4, 1, DEV, 4, 0, DEV), -9),
    ((DEV, 4, 4, DEV, 4, 1, DEV, 4, DEV, 0), -12),
])
def test_dispatch_solve_argument_checks(args, expect):
    rc, _, _ = bandlu.dispatch_solve(*args, stream=0)
    assert rc == expect


def test_binding_has_the_c_names():
    for name in declared_functions():
        if name == "bandlu_version":
            continue
        assert callable(getattr(bandlu, name)), name


@pytest.mark.parametrize("args,expect", [
    ((2, 4, 1, DEV, 4, DEV, 4, 1, DEV), -1),
    ((1, -1, 1, DEV, 4, DEV, 4, 1, DEV), -2),
    ((1, 4, -1, DEV, 4, DEV, 4, 1, DEV), -3),
    ((1, 4, 4, DEV, 4, DEV, 4, 1, DEV), -3),
    ((1, 4, 1, 0, 4, DEV, 4, 1, DEV), -4),
    ((0, 4, 1, DEV, 3, DEV, 4, 1, DEV), -5),
    ((1, 4, 1, DEV, 4, 0, 4, 1, DEV), -6),
    ((1, 4, 1, DEV, 4, DEV, 3, 1, DEV), -7),
    ((1, 4, 1, DEV, 4, DEV, 4, -1, DEV), -8),
    ((1, 4, 1, DEV, 4, DEV, 4, 1, 0), -9),
])
def test_trsv_band_argument_checks(args, expect):
    assert bandlu.trsv_band(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((-1, DEV, 4, DEV, 4, 1, DEV), -1),
    ((4, 0, 4, DEV, 4, 1, DEV), -2),
    ((4, DEV, 3, DEV, 4, 1, DEV), -3),
    ((4, DEV, 4, 0, 4, 1, DEV), -4),
    ((4, DEV, 4, DEV, 3, 1, DEV), -5),
    ((4, DEV, 4, DEV, 4, -1, DEV), -6),
    ((4, DEV, 4, DEV, 4, 1, 0), -7),
])
def test_diag_solve_argument_checks(args, expect):
    assert bandlu.diag_solve(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, DEV, 4, 1, DEV, 4, DEV, DEV), -1),
    ((DEV, -2, 4, DEV, 4, 1, DEV, 4, DEV, DEV), -2),
    ((DEV, 4, 3, DEV, 4, 1, DEV, 4, DEV, DEV), -3),
    ((DEV, 4, 4, 0, 4, 1, DEV, 4, DEV, DEV), -4),
    ((DEV, 4, 4, DEV, 3, 1, DEV, 4, DEV, DEV), -5),
    ((DEV, 4, 4, DEV, 4, -1, DEV, 4, DEV, DEV), -6),
    ((DEV, 4, 4, DEV, 4, 1, 0, 4, DEV, DEV), -7),
    ((DEV, 4, 4, DEV, 4, 1, DEV, 0, DEV, DEV), -8),
    ((DEV, 4, 4, DEV, 4, 1, DEV, 4, 0, DEV), -9),
    ((DEV, 4, 4, DEV, 4, 1, DEV, 4, DEV, 0), -13),
])
def test_dispatch_backslash_argument_checks(args, expect):
    rc, _, _, _ = bandlu.dispatch_backslash(*args, stream=0)
    assert rc == expect


def test_classify_matches_the_oracle(oracle_mod):
    """The host-side branch choice of the backslash dispatch agrees with the oracle's."""
    import itertools
    assert bandlu.bandlu_classify(4, -1, 0, 4) == -1
    for n, kl, ku, ldab in itertools.product([0, 1, 2, 7, 64, 1000, 1 << 20], [0, 1, 3, 30, 999],
                                             [0, 1, 2, 64, 500], [1, 4, 10, 200, 4000]):
        if n and (kl > n - 1 or ku > n - 1):
            continue
        assert bandlu.bandlu_classify(n, kl, ku, ldab) == oracle_mod.classify(n, kl, ku, ldab), (n, kl, ku, ldab)


def test_classify_at_the_hand_worked_thresholds():
    """The library's predicate at the smallest n that takes the band path, worked by hand
    from the paper's operation counts (tests/golden/predicate_threshold_cases.txt)."""
    path = os.path.join(ROOT, "tests", "golden", "predicate_threshold_cases.txt")
    rows = [tuple(int(x) for x in ln.split()) for ln in open(path) if ln.strip() and not ln.startswith("#")]
    assert len(rows) == 7
    for kl, ku, n_min in rows:
        if kl == 0 or ku == 0:
            continue  # the diagonal and triangular branches come first there
        ldab = 2 * kl + ku + 1
        assert bandlu.bandlu_classify(n_min, kl, ku, ldab) == bandlu.KIND_BANDED, (kl, ku, n_min)
        assert bandlu.bandlu_classify(n_min - 1, kl, ku, ldab) == bandlu.KIND_DENSE, (kl, ku, n_min)


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, DEV, 4, DEV, DEV, DEV, DEV, DEV), -1),
    ((DEV, -2, 4, DEV, 4, DEV, DEV, DEV, DEV, DEV), -2),
    ((DEV, 4, 3, DEV, 4, DEV, DEV, DEV, DEV, DEV), -3),
    ((DEV, 4, 4, 0, 4, DEV, DEV, DEV, DEV, DEV), -4),
    ((DEV, 4, 4, DEV, 0, DEV, DEV, DEV, DEV, DEV), -5),
    ((DEV, 4, 4, DEV, 4, 0, DEV, DEV, DEV, DEV), -6),
    ((DEV, 4, 4, DEV, 4, DEV, 0, DEV, DEV, DEV), -7),
    ((DEV, 4, 4, DEV, 4, DEV, DEV, 0, DEV, DEV), -8),
    ((DEV, 4, 4, DEV, 4, DEV, DEV, DEV, 0, DEV), -9),
    ((DEV, 4, 4, DEV, 4, DEV, DEV, DEV, DEV, 0), -10),
])
def test_dispatch_lu_async_argument_checks(args, expect):
    assert bandlu.dispatch_lu_async(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((DEV, -1, 1, DEV, DEV), -2), ((0, 4, 4, DEV, DEV), -1), ((DEV, 4, 3, DEV, DEV), -3),
    ((DEV, 4, 4, 0, DEV), -4), ((DEV, 4, 4, DEV, 0), -5),
])
def test_detect_bandwidth_cm_argument_checks(args, expect):
    assert bandlu.detect_bandwidth_cm(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, 1, 1, DEV, 4), -1), ((DEV, 3, 4, 1, 1, DEV, 4), -2), ((DEV, 4, -1, 1, 1, DEV, 4), -3),
    ((DEV, 4, 4, -1, 1, DEV, 4), -4), ((DEV, 4, 4, 1, -1, DEV, 4), -5), ((DEV, 4, 4, 1, 1, 0, 4), -6),
    ((DEV, 4, 4, 1, 1, DEV, 3), -7),
])
def test_dense_to_band_cm_argument_checks(args, expect):
    assert bandlu.dense_to_band_cm(*args, stream=0) == expect


@pytest.mark.parametrize("args,expect", [
    ((0, 4, 4, DEV, 4, DEV, DEV), -1), ((DEV, -2, 4, DEV, 4, DEV, DEV), -2), ((DEV, 4, 2, DEV, 4, DEV, DEV), -3),
    ((DEV, 4, 4, 0, 4, DEV, DEV), -4), ((DEV, 4, 4, DEV, 0, DEV, DEV), -5), ((DEV, 4, 4, DEV, 4, 0, DEV), -6),
    ((DEV, 4, 4, DEV, 4, DEV, 0), -9),
])
def test_dispatch_lu_cm_argument_checks(args, expect):
    rc, _, _ = bandlu.dispatch_lu_cm(*args, stream=0)
    assert rc == expect


BIG = 1 << 62  # a leading dimension or stride whose extent over the matrix would overflow 64 bits


@pytest.mark.parametrize("call,expect", [
    (lambda: bandlu.detect_bandwidth(DEV, 4, BIG, DEV, DEV, stream=0), -3),
    (lambda: bandlu.dense_to_band(DEV, BIG, 4, 1, 1, DEV, 4, stream=0), -2),
    (lambda: bandlu.dense_to_band(DEV, 4, 4, 1, 1, DEV, BIG, stream=0), -7),
    (lambda: bandlu.gbtrf(4, 1, 1, DEV, BIG, DEV, DEV, stream=0), -5),
    (lambda: bandlu.gbtrs(4, 1, 1, 8, DEV, 4, DEV, DEV, BIG, stream=0), -9),
    (lambda: bandlu.dispatch_lu(DEV, 4, BIG, DEV, 4, DEV, DEV, stream=0)[0], -3),
    (lambda: bandlu.dispatch_lu_noalloc(DEV, 4, BIG, DEV, 4, DEV, DEV, stream=0)[0], -3),
    (lambda: bandlu.dispatch_lu_noalloc(DEV, 4, 4, DEV, BIG, DEV, DEV, stream=0)[0], -5),
    (lambda: bandlu.dispatch_lu_batched(DEV, 4, 4, BIG, 8, DEV, 4, 16, DEV, 4, DEV, DEV, DEV, DEV, stream=0), -4),
    (lambda: bandlu.dispatch_lu_batched(DEV, 4, 4, 16, 8, DEV, 4, BIG, DEV, 4, DEV, DEV, DEV, DEV, stream=0), -8),
    (lambda: bandlu.trsv_band(1, 4, 1, DEV, 4, DEV, BIG, 8, DEV, stream=0), -7),
])
def test_overflowing_extents_are_rejected(call, expect):
    assert call() == expect


def test_peak_microbenchmarks_reject_bad_arguments():
    # the argument checks run on the host before any launch (stream 0: no CUDA call)
    assert bandlu.bandlu_peak_warp_costs(8, DEV, DEV, 1, 1, 0) == -1
    assert bandlu.bandlu_peak_warp_costs(-1, DEV, DEV, 1, 1, 0) == -1
    assert bandlu.bandlu_peak_warp_costs(0, 0, DEV, 1, 1, 0) == -2
    assert bandlu.bandlu_peak_warp_costs(0, DEV, 0, 1, 1, 0) == -3
    assert bandlu.bandlu_peak_warp_costs(0, DEV, DEV, 0, 1, 0) == -4
    assert bandlu.bandlu_peak_warp_costs(0, DEV, DEV, 33, 1, 0) == -4
    assert bandlu.bandlu_peak_warp_costs(0, DEV, DEV, 1, 0, 0) == -5
    assert bandlu.bandlu_peak_dfma(0, 1, 32, 1, 1, 0) == -1
    assert bandlu.bandlu_peak_dfma(DEV, 1, 48, 1, 1, 0) == -3
    assert bandlu.bandlu_peak_dfma(DEV, 1, 32, 9, 1, 0) == -4
    assert bandlu.bandlu_peak_dmma(2, DEV, 1, 1, 1, 1, 0) == -1
    assert bandlu.bandlu_peak_dmma(0, DEV, 1, 1, 5, 1, 0) == -5
    assert bandlu.bandlu_peak_hbm_read(DEV + 8, 64, DEV, 1, 0) == -1
    assert bandlu.bandlu_peak_hbm_read(DEV, 24, DEV, 1, 0) == -2
