"""The integer-pipe reciprocal on the pivot chain must be IEEE round-to-nearest
division bit for bit (the multipliers are a * (1/pivot), the DGBTF2 form).
Host copy of the same code against numpy's division (CPU); device copy against
the GPU's own double division and numpy (GPU)."""
import numpy as np
import pytest

from paper_2608_22099_gb300 import bandlu


def edge_inputs():
    fr = [0, 1, 2, 3, (1 << 52) - 1, (1 << 52) - 2, 1 << 51, (1 << 51) + 1, (1 << 51) - 1]
    fr += [(1 << 52) - (1 << k) for k in range(52)] + [1 << k for k in range(52)]
    fr += [(1 << k) + 1 for k in range(52)] + [(1 << k) - 1 for k in range(1, 52)]
    fr = np.array(fr, dtype=np.int64)
    ex = np.arange(0, 2048, dtype=np.int64)
    x = ((ex[:, None] << 52) | fr[None, :]).reshape(-1).view(np.float64)
    return np.concatenate([x, -x])


def random_inputs(n, seed):
    rng = np.random.default_rng(seed)
    a = rng.integers(0, 2 ** 63, n, dtype=np.int64).view(np.float64)
    b = rng.standard_normal(n) * np.exp(rng.uniform(-700, 700, n))
    m = rng.integers(1 << 52, 1 << 53, n, dtype=np.int64)
    c = ((np.int64(1023) << 52) | (m & ((1 << 52) - 1))).view(np.float64)
    specials = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, 2.2250738585072014e-308,
                         1.7976931348623157e308, 2.0 ** 1021, 2.0 ** 1020 * 1.5, 2.0 ** -1022])
    return np.concatenate([a, b, c, specials])


def same_bits(y, ref):
    return (y.view(np.int64) == ref.view(np.int64)) | (np.isnan(y) & np.isnan(ref))


@pytest.mark.parametrize("source", ["edge", "random"])
def test_reciprocal_host_copy_is_ieee_division(source):
    x = edge_inputs() if source == "edge" else random_inputs(1_000_000, 3)
    x = np.ascontiguousarray(x)
    y = np.empty_like(x)
    bandlu.bandlu_selftest_rcp_host(x, y, x.size)
    with np.errstate(all="ignore"):
        ref = 1.0 / x
    bad = ~same_bits(y, ref)
    assert not bad.any(), x[bad][:5]


@pytest.mark.gpu
@pytest.mark.parametrize("source", ["edge", "random"])
def test_reciprocal_device_is_ieee_division(source):
    import torch
    x = edge_inputs() if source == "edge" else random_inputs(4_000_000, 11)
    xd = torch.from_numpy(np.ascontiguousarray(x)).cuda()
    y = torch.empty_like(xd)
    yd = torch.empty_like(xd)
    assert bandlu.bandlu_selftest_rcp_device(xd, y, x.size, 0) == 0
    assert bandlu.bandlu_selftest_rcp_device(xd, yd, x.size, 1) == 0
    torch.cuda.synchronize()
    y, yd = y.cpu().numpy(), yd.cpu().numpy()
    with np.errstate(all="ignore"):
        ref = 1.0 / x
    assert same_bits(y, yd).all(), x[~same_bits(y, yd)][:5]
    assert same_bits(y, ref).all(), x[~same_bits(y, ref)][:5]
