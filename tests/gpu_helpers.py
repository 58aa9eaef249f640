"""Shared helpers of the GPU parity tests: run each entry point through the C ABI
on device tensors and bring the results back for comparison with the oracle."""
import numpy as np
import torch

from paper_2608_22099_gb300 import bandlu

DEV = "cuda:0"


def detect_gpu(A_dev: torch.Tensor, n: int | None = None, lda: int | None = None):
    n = A_dev.shape[0] if n is None else n
    lda = A_dev.shape[1] if lda is None else lda
    out = torch.full((2,), -7, dtype=torch.int32, device=A_dev.device)
    rc = bandlu.detect_bandwidth(A_dev, n, lda, out, out.data_ptr() + 4)
    torch.cuda.synchronize()
    assert rc == 0, rc
    kl, ku = out.tolist()
    return kl, ku


def convert_gpu(A_dev: torch.Tensor, kl: int, ku: int, ldab: int, fill: float = np.nan):
    n, lda = A_dev.shape[0], A_dev.shape[1]
    AB = torch.full((n, ldab), fill, dtype=torch.float64, device=A_dev.device)
    rc = bandlu.dense_to_band(A_dev, lda, n, kl, ku, AB, ldab)
    torch.cuda.synchronize()
    assert rc == 0, rc
    return AB


def gbtrf_gpu(AB_host: np.ndarray, kl: int, ku: int):
    """Factor a copy of the (n, ldab) band on the GPU; returns (AB, ipiv, info) on the host."""
    n, ldab = AB_host.shape
    AB = torch.from_numpy(np.ascontiguousarray(AB_host)).to(DEV)
    ipiv = torch.full((max(n, 1),), -1, dtype=torch.int32, device=DEV)
    info = torch.full((1,), -5, dtype=torch.int32, device=DEV)
    rc = bandlu.gbtrf(n, kl, ku, AB, ldab, ipiv, info)
    torch.cuda.synchronize()
    assert rc == 0, rc
    return AB.cpu().numpy(), ipiv.cpu().numpy()[:n], int(info.item())


def rel_diff(a: np.ndarray, b: np.ndarray) -> float:
    scale = float(np.max(np.abs(b))) if b.size else 0.0
    d = float(np.max(np.abs(a - b))) if a.size else 0.0
    return d / scale if scale > 0 else d


def assert_factor_parity(AB_gpu, ipiv_gpu, info_gpu, AB_ref, ipiv_ref, info_ref, tol=1e-12, bitwise=True):
    """Integers bit-exact; factors within tol relative (inf-norm over all entries);
    optionally bit-identical (the kernels follow the oracle's order of operations)."""
    assert info_gpu == info_ref, (info_gpu, info_ref)
    if not np.array_equal(ipiv_gpu, ipiv_ref):
        j = int(np.argmax(ipiv_gpu != ipiv_ref))
        raise AssertionError(f"ipiv differs first at column {j}: gpu {ipiv_gpu[j]} oracle {ipiv_ref[j]}")
    assert rel_diff(AB_gpu, AB_ref) <= tol, rel_diff(AB_gpu, AB_ref)
    if bitwise:
        same = AB_gpu.view(np.int64) == AB_ref.view(np.int64)
        if not np.all(same):
            j, r = np.argwhere(~same)[0]
            raise AssertionError(f"AB not bit-identical first at column {j} row {r}: {AB_gpu[j, r]!r} vs {AB_ref[j, r]!r}")
