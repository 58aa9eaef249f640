"""Seeded synthetic inputs: banded fp64 matrices stored dense.

This module holds input construction only (none of the method's arithmetic):
it draws the in-band values from a seeded torch CPU generator and scatters them
into a zeroed dense row-major matrix.  The same draw serves the CUDA path
(scattered on the device) and the CPU oracle (scattered on the host), so both
see bit-identical inputs.

Recipe (the paper draws random banded matrices but states no distribution,
Sec. IV-A; these stand in for them):
  * values are drawn as an array of shape (n, kl+ku+1) [or (batch, n, kl+ku+1)],
    entry (i, d) belonging to element (i, j = i + d - kl); entries whose column
    falls outside 0..n-1 are drawn and dropped;
  * "uniform" is 2*U[0,1) - 1, "normal" is N(0, 1);
  * an optional constant is added to the diagonal (diagonal dominance);
  * everything outside the band is an exact +0.0.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: n x n banded matrix (or a batch of them) stored dense."""
    name: str
    n: int
    kl: int
    ku: int
    dist: str          # "uniform" or "normal"
    diag_boost: float
    seed: int
    batch: int = 0     # 0: a single matrix
    stray: tuple = ()  # optional (i, j, value) placed after the band (control input)
    notes: str = field(default="", compare=False)

    @property
    def ldab(self) -> int:
        return 2 * self.kl + self.ku + 1


# The five workload shapes the benchmark and the tests use.
WORKLOADS = {
    "n512_kl3_ku3": Workload("n512_kl3_ku3", 512, 3, 3, "uniform", 12.0, 1001,
                             notes="diagonally dominant: pivots stay on the diagonal"),
    "n4096_kl16_ku16": Workload("n4096_kl16_ku16", 4096, 16, 16, "uniform", 0.0, 1002,
                                notes="no diagonal boost: partial pivoting swaps rows"),
    "n16384_kl8_ku64": Workload("n16384_kl8_ku64", 16384, 8, 64, "normal", 0.0, 1003),
    "n16384_kl8_ku64_stray": Workload("n16384_kl8_ku64_stray", 16384, 8, 64, "normal", 0.0, 1003,
                                      stray=(16383, 0, 1e-3),
                                      notes="control: one stray entry makes kl = n-1 (not banded)"),
    "batch4096_n256_kl2_ku2": Workload("batch4096_n256_kl2_ku2", 256, 2, 2, "uniform", 4.0, 1004, batch=4096),
    "n32768_kl256_ku256": Workload("n32768_kl256_ku256", 32768, 256, 256, "uniform", 0.0, 1005),
}


def band_values(n: int, kl: int, ku: int, dist: str, seed: int, batch: int = 0) -> torch.Tensor:
    """Seeded in-band values, float64 on the CPU, shape ([batch,] n, kl+ku+1)."""
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    shape = (n, kl + ku + 1) if batch == 0 else (batch, n, kl + ku + 1)
    if dist == "uniform":
        return 2.0 * torch.rand(shape, generator=g, dtype=torch.float64) - 1.0
    if dist == "normal":
        return torch.randn(shape, generator=g, dtype=torch.float64)
    raise ValueError(f"unknown distribution {dist!r}")


def scatter_band(A: torch.Tensor, vals: torch.Tensor, kl: int, ku: int, diag_boost: float = 0.0) -> torch.Tensor:
    """Write the band values into the (zeroed) dense matrix A[..., :n, :n] in place."""
    n = vals.shape[-2]
    M = A[..., :n, :n]
    vals = vals.to(A.device)
    for d in range(-kl, ku + 1):
        if abs(d) >= n:
            continue
        rows = slice(max(0, -d), min(n, n - d))
        v = vals[..., rows, d + kl]
        if d == 0 and diag_boost != 0.0:
            v = v + diag_boost
        M.diagonal(offset=d, dim1=-2, dim2=-1).copy_(v)
    return A


def make_dense(n: int, kl: int, ku: int, *, dist: str = "uniform", diag_boost: float = 0.0, seed: int = 0,
               batch: int = 0, lda: int | None = None, device: str | torch.device = "cpu",
               stray: tuple = ()) -> torch.Tensor:
    """Dense row-major storage ([batch,] n, lda) of a seeded banded matrix (zeros outside the band)."""
    lda = n if lda is None else lda
    shape = (n, lda) if batch == 0 else (batch, n, lda)
    A = torch.zeros(shape, dtype=torch.float64, device=device)
    if n == 0:
        return A
    vals = band_values(n, kl, ku, dist, seed, batch)
    scatter_band(A, vals, kl, ku, diag_boost)
    if stray:
        i, j, v = stray
        A[..., i, j] = v
    return A


def make_workload(w: Workload, device: str | torch.device = "cpu", lda: int | None = None) -> torch.Tensor:
    return make_dense(w.n, w.kl, w.ku, dist=w.dist, diag_boost=w.diag_boost, seed=w.seed, batch=w.batch,
                      lda=lda, device=device, stray=w.stray)


def principal_block(w: Workload, m: int) -> torch.Tensor:
    """The leading m x m principal block of workload w's matrix, built on the host without
    the full matrix: the same seeded draw, scattered for rows 0..m-1 with the columns beyond
    m-1 dropped.  A principal block of a banded matrix is banded with the same (kl, ku)."""
    if w.batch:
        raise ValueError("principal_block takes a single-matrix workload")
    m = min(m, w.n)
    vals = band_values(w.n, w.kl, w.ku, w.dist, w.seed)[:m]
    A = torch.zeros((m, m), dtype=torch.float64)
    scatter_band(A, vals, w.kl, w.ku, w.diag_boost)
    if w.stray and w.stray[0] < m and w.stray[1] < m:
        A[w.stray[0], w.stray[1]] = w.stray[2]
    return A
