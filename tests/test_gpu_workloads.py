"""Parity at the full workload sizes, in the launch configuration the benchmark times:
dispatch_lu (or dispatch_lu_batched) through the C ABI against the CPU oracle on the
whole problem.  Integers bit-exact, factors within 1e-12 relative, backward error
<= 10 in units of n * eps * ||A||."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import DEV, assert_factor_parity
from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300.workloads import WORKLOADS, make_workload

pytestmark = pytest.mark.gpu

SINGLE = ["n512_kl3_ku3", "n4096_kl16_ku16", "n16384_kl8_ku64", "n32768_kl256_ku256"]


@pytest.mark.parametrize("name", SINGLE)
def test_workload_dispatch_lu(name):
    w = WORKLOADS[name]
    A = make_workload(w)                       # host copy for the oracle
    Ad = A.to(DEV)
    n, ldab = w.n, w.ldab
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=DEV)
    ipiv = torch.zeros(n, dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, kl, ku = bandlu.dispatch_lu(Ad, n, n, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    del Ad
    An = A.numpy()
    okl, oku = oracle.detect_bandwidth(An)
    assert (rc, kl, ku) == (0, okl, oku) == (0, w.kl, w.ku)
    ABo = oracle.dense_to_band(An, kl, ku, ldab)
    ABf, ipiv_o, info_o, _ = oracle.gbtrf(ABo, kl, ku)
    got_AB, got_ipiv = AB.cpu().numpy(), ipiv.cpu().numpy()
    assert_factor_parity(got_AB, got_ipiv, int(info.item()), ABf, ipiv_o, info_o)
    assert oracle.backward_error(An, got_AB, got_ipiv, kl, ku) <= 10.0
    # the solve with these factors, one right-hand side, bit-identical to the oracle's
    b = np.linspace(-1.0, 1.0, n)
    xd = torch.from_numpy(b.copy()).to(DEV)
    assert bandlu.gbtrs(n, kl, ku, 1, AB, ldab, ipiv, xd, n) == 0
    torch.cuda.synchronize()
    x_ref = oracle.gbtrs(ABf, ipiv_o, kl, ku, b[None])[0]
    x = xd.cpu().numpy()
    # back substitution can overflow on these random bands (n = 16384, kl = 8); infinities must
    # match bit for bit, NaNs in position (their payloads are the platform's)
    nan_g, nan_r = np.isnan(x), np.isnan(x_ref)
    assert np.array_equal(nan_g, nan_r)
    assert np.array_equal(x[~nan_g].view(np.int64), x_ref[~nan_r].view(np.int64))


def test_workload_stray_entry_control():
    w = WORKLOADS["n16384_kl8_ku64_stray"]
    A = make_workload(w)
    Ad = A.to(DEV)
    n = w.n
    AB = torch.full((n, w.ldab), -3.0, dtype=torch.float64, device=DEV)
    ipiv = torch.full((n,), -1, dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, kl, ku = bandlu.dispatch_lu(Ad, n, n, AB, w.ldab, ipiv, info)
    torch.cuda.synchronize()
    assert (rc, kl, ku) == (bandlu.BANDLU_NOT_BANDED, n - 1, w.ku)
    assert oracle.detect_bandwidth(A.numpy()) == (kl, ku)
    assert not oracle.is_banded(n, kl, ku, w.ldab)
    assert bool(torch.all(AB == -3.0)) and bool(torch.all(ipiv == -1)) and int(info.item()) == -5


def test_workload_batched():
    w = WORKLOADS["batch4096_n256_kl2_ku2"]
    A = make_workload(w)
    Ad = A.to(DEV)
    B, n, ldab = w.batch, w.n, w.ldab
    AB = torch.zeros((B, n, ldab), dtype=torch.float64, device=DEV)
    ipiv = torch.zeros((B, n), dtype=torch.int32, device=DEV)
    kl, ku, info, status = (torch.full((B,), -1, dtype=torch.int32, device=DEV) for _ in range(4))
    rc = bandlu.dispatch_lu_batched(Ad, n, n, n * n, B, AB, ldab, n * ldab, ipiv, n, kl, ku, info, status)
    torch.cuda.synchronize()
    assert rc == 0
    ref = oracle.dispatch_lu_batched(A.numpy(), ldab)
    for key, t in (("kl", kl), ("ku", ku), ("info", info), ("status", status)):
        assert np.array_equal(t.cpu().numpy(), ref[key]), key
    assert np.all(ref["status"] == 0) and np.all(ref["kl"] == 2) and np.all(ref["ku"] == 2)
    got_AB, got_ipiv = AB.cpu().numpy(), ipiv.cpu().numpy()
    assert np.array_equal(got_ipiv, ref["ipiv"])
    scale = np.max(np.abs(ref["AB"]), axis=(1, 2))
    rel = np.max(np.abs(got_AB - ref["AB"]), axis=(1, 2)) / scale
    assert float(np.max(rel)) <= 1e-12
    assert np.array_equal(got_AB.view(np.int64), ref["AB"].view(np.int64))
    An = A.numpy()
    for b in range(0, B, 97):
        assert oracle.backward_error(An[b], got_AB[b], got_ipiv[b], 2, 2) <= 10.0
