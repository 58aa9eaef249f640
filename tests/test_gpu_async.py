"""GPU parity of dispatch_lu_async (the dispatch decision taken on the device, no host
synchronisation) against the oracle and against dispatch_lu, and its capture in a CUDA
graph replayed on new inputs."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import DEV
from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300.workloads import make_dense

pytestmark = pytest.mark.gpu


class AsyncOut:
    def __init__(self, n, ldab):
        self.AB = torch.full((max(n, 1), ldab), -3.0, dtype=torch.float64, device=DEV)
        self.ipiv = torch.full((max(n, 1),), -1, dtype=torch.int32, device=DEV)
        self.sc = torch.full((4,), -7, dtype=torch.int32, device=DEV)  # kl, ku, status, info

    def call(self, Ad, n, lda, ldab):
        s = self.sc
        return bandlu.dispatch_lu_async(Ad, n, lda, self.AB, ldab, self.ipiv, s[0:1], s[1:2], s[2:3], s[3:4])

    def result(self):
        kl, ku, status, info = (int(v) for v in self.sc.cpu())
        return kl, ku, status, info, self.AB.cpu().numpy(), self.ipiv.cpu().numpy()


def check_against_oracle(A, ldab, out):
    n = A.shape[0]
    kl, ku, status, info, AB, ipiv = out.result()
    r = oracle.dispatch_lu(A, ldab)
    assert (kl, ku, status) == (r["kl"], r["ku"], r["status"])
    if status == 0:
        assert info == r["info"]
        assert np.array_equal(ipiv[:n], r["ipiv"])
        assert np.array_equal(AB[:n].view(np.int64), r["AB"].view(np.int64))
    else:
        assert info == -7 and np.all(AB == -3.0) and np.all(ipiv == -1)


# register window, shared-memory windows of several shapes, the block-wide generic path
# (kl > 27), declined (capacity, predicate), degenerate sizes
@pytest.mark.parametrize("n,kl,ku,ldab,boost", [(1, 0, 0, 1, 1.0), (2, 1, 0, 3, 0.0), (512, 3, 3, 10, 12.0),
                                                (512, 3, 3, 40, 0.0), (4096, 16, 16, 49, 0.0),
                                                (3000, 8, 64, 81, 0.0), (2000, 27, 100, 256, 0.0),
                                                (1500, 40, 40, 121, 0.0), (800, 2, 2, 4, 0.0),
                                                (60, 50, 50, 151, 0.0), (0, 0, 0, 1, 0.0)])
def test_dispatch_lu_async_matches_oracle(n, kl, ku, ldab, boost):
    A = make_dense(n, kl, ku, dist="uniform", diag_boost=boost, seed=n + kl + ku).numpy()
    out = AsyncOut(n, ldab)
    Ad = torch.from_numpy(A).to(DEV)
    assert out.call(Ad, n, max(n, 1), ldab) == 0
    torch.cuda.synchronize()
    check_against_oracle(A, ldab, out)


def test_dispatch_lu_async_equals_dispatch_lu():
    n, kl, ku = 4096, 16, 16
    ldab = 2 * kl + ku + 1
    A = make_dense(n, kl, ku, dist="uniform", diag_boost=0.0, seed=1002)
    Ad = A.to(DEV)
    out = AsyncOut(n, ldab)
    assert out.call(Ad, n, n, ldab) == 0
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=DEV)
    ipiv = torch.zeros(n, dtype=torch.int32, device=DEV)
    info = torch.zeros(1, dtype=torch.int32, device=DEV)
    rc, gkl, gku = bandlu.dispatch_lu(Ad, n, n, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    kl2, ku2, status, info2, AB2, ipiv2 = out.result()
    assert (rc, gkl, gku, int(info.item())) == (status, kl2, ku2, info2)
    assert torch.equal(ipiv.cpu(), torch.from_numpy(ipiv2))
    assert np.array_equal(AB.cpu().numpy().view(np.int64), AB2.view(np.int64))


def test_dispatch_lu_async_in_a_cuda_graph():
    """Captured once, replayed on three different matrices copied into the same input buffer:
    each replay detects, decides and factors anew on the device."""
    n, ldab = 1024, 40
    mats = [make_dense(n, 3, 3, dist="uniform", diag_boost=0.0, seed=11).numpy(),
            make_dense(n, 9, 12, dist="uniform", diag_boost=0.0, seed=12).numpy(),
            make_dense(n, 2, 30, dist="uniform", diag_boost=0.0, seed=13).numpy()]
    mats[2][n - 1, 0] = 1e-3  # declined: kl = n-1
    Ad = torch.zeros((n, n), dtype=torch.float64, device=DEV)
    out = AsyncOut(n, ldab)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        assert out.call(Ad, n, n, ldab) == 0  # warm-up outside the capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        rc = out.call(Ad, n, n, ldab)
    assert rc == 0
    for A in mats:
        out.AB.fill_(-3.0)
        out.ipiv.fill_(-1)
        out.sc.fill_(-7)
        Ad.copy_(torch.from_numpy(A))
        g.replay()
        torch.cuda.synchronize()
        check_against_oracle(A, ldab, out)


@pytest.mark.parametrize("n,kl,ku,ldab", [(2049, 256, 256, 769), (1200, 40, 30, 111), (3000, 100, 20, 221)])
def test_dispatch_lu_async_wide_bands(n, kl, ku, ldab):
    """Wide bands: the multi-CTA cluster kernel, enqueued before the bandwidths are known, takes
    them on the device; bit-identical to dispatch_lu (which chose the same kernel on the host)
    and to the oracle."""
    A = make_dense(n, kl, ku, dist="uniform", diag_boost=0.0, seed=n + 7 * kl).numpy()
    out = AsyncOut(n, ldab)
    Ad = torch.from_numpy(A).to(DEV)
    assert out.call(Ad, n, n, ldab) == 0
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=DEV)
    ipiv = torch.zeros(n, dtype=torch.int32, device=DEV)
    info = torch.zeros(1, dtype=torch.int32, device=DEV)
    rc, gkl, gku = bandlu.dispatch_lu(Ad, n, n, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    kl2, ku2, status, info2, AB2, ipiv2 = out.result()
    assert (rc, gkl, gku, int(info.item())) == (status, kl2, ku2, info2) == (0, kl, ku, 0)
    assert np.array_equal(AB.cpu().numpy().view(np.int64), AB2.view(np.int64))
    assert torch.equal(ipiv.cpu(), torch.from_numpy(ipiv2))
    check_against_oracle(A, ldab, out)


def test_dispatch_lu_async_wide_band_in_a_cuda_graph():
    """One capture with band storage that admits wide bands, replayed on a wide band (the
    multi-CTA kernel), a narrow one (register window), a windowed one and a declined one."""
    n, ldab = 1500, 121
    mats = [make_dense(n, 40, 30, dist="uniform", diag_boost=0.0, seed=21).numpy(),
            make_dense(n, 3, 3, dist="uniform", diag_boost=0.0, seed=22).numpy(),
            make_dense(n, 20, 50, dist="uniform", diag_boost=0.0, seed=23).numpy(),
            make_dense(n, 50, 20, dist="uniform", diag_boost=0.0, seed=24).numpy()]
    mats[3][n - 1, 0] = 1e-3  # declined: kl = n-1
    Ad = torch.zeros((n, n), dtype=torch.float64, device=DEV)
    out = AsyncOut(n, ldab)
    s = torch.cuda.Stream()
    Ad.copy_(torch.from_numpy(mats[0]))
    with torch.cuda.stream(s):
        assert out.call(Ad, n, n, ldab) == 0  # warm-up outside the capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        rc = out.call(Ad, n, n, ldab)
    assert rc == 0
    for A in mats:
        out.AB.fill_(-3.0)
        out.ipiv.fill_(-1)
        out.sc.fill_(-7)
        Ad.copy_(torch.from_numpy(A))
        g.replay()
        torch.cuda.synchronize()
        check_against_oracle(A, ldab, out)
