"""GPU parity of the column-major entry points (element (i, j) at A[i + j*lda]) against the
oracle: bandwidths and pivots bit for bit, band storage and factors bit-identical."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import DEV
from paper_2608_22099_gb300 import bandlu
from paper_2608_22099_gb300.workloads import make_dense

pytestmark = pytest.mark.gpu


def column_major(M, pad=3):
    n = M.shape[0]
    Acm = np.full((n, n + pad), np.nan)  # the padding is never read
    Acm[:, :n] = M.T
    return Acm


@pytest.mark.parametrize("n,kl,ku", [(1, 0, 0), (2, 0, 1), (17, 3, 5), (512, 3, 3), (1000, 90, 7), (4096, 16, 16)])
def test_detect_and_convert_cm_match_oracle(n, kl, ku):
    M = make_dense(n, kl, ku, dist="uniform", diag_boost=0.0, seed=n + kl).numpy()
    Acm = column_major(M)
    assert oracle.detect_bandwidth_cm(Acm) == (kl, ku)
    Ad = torch.from_numpy(Acm).to(DEV)
    out = torch.full((2,), -1, dtype=torch.int32, device=DEV)
    assert bandlu.detect_bandwidth_cm(Ad, n, Acm.shape[1], out[0:1], out[1:2]) == 0
    torch.cuda.synchronize()
    assert tuple(int(v) for v in out.cpu()) == (kl, ku)
    ldab = 2 * kl + ku + 2
    AB = torch.full((n, ldab), 7.0, dtype=torch.float64, device=DEV)
    assert bandlu.dense_to_band_cm(Ad, Acm.shape[1], n, kl, ku, AB, ldab) == 0
    torch.cuda.synchronize()
    ref = oracle.dense_to_band_cm(Acm, kl, ku, ldab)
    assert np.array_equal(AB.cpu().numpy().view(np.int64), ref.view(np.int64))


@pytest.mark.parametrize("n,kl,ku,ldab", [(512, 3, 3, 10), (4096, 16, 16, 49), (3000, 40, 20, 101), (800, 2, 2, 6)])
def test_dispatch_lu_cm_matches_oracle(n, kl, ku, ldab):
    M = make_dense(n, kl, ku, dist="uniform", diag_boost=0.0, seed=3 * n + ku).numpy()
    Acm = column_major(M, pad=0)
    Ad = torch.from_numpy(Acm).to(DEV)
    AB = torch.full((n, ldab), -3.0, dtype=torch.float64, device=DEV)
    ipiv = torch.full((n,), -1, dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc, gkl, gku = bandlu.dispatch_lu_cm(Ad, n, n, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    r = oracle.dispatch_lu(M, ldab)  # the same matrix, row-major, through the row-major oracle
    assert (rc, gkl, gku) == (r["status"], r["kl"], r["ku"])
    if rc == 0:
        assert int(info.item()) == r["info"]
        assert np.array_equal(ipiv.cpu().numpy(), r["ipiv"])
        assert np.array_equal(AB.cpu().numpy().view(np.int64), r["AB"].view(np.int64))
    else:
        assert int(info.item()) == -5
