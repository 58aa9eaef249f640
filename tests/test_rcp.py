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


def division_pairs(n, seed):
    """Dividend/divisor pairs: random bit patterns, wide-range normals, equal
    exponents, exact quotients (x = d*m with short m), quotients whose last bits
    lie near a rounding midpoint, and every class of special value on either side."""
    rng = np.random.default_rng(seed)
    k = n // 6
    x1 = rng.integers(0, 2 ** 63, k, dtype=np.int64).view(np.float64)
    d1 = rng.integers(0, 2 ** 63, k, dtype=np.int64).view(np.float64)
    x2 = rng.standard_normal(k) * np.exp(rng.uniform(-300, 300, k))
    d2 = rng.standard_normal(k) * np.exp(rng.uniform(-300, 300, k))
    x3 = rng.uniform(1.0, 2.0, k)
    d3 = rng.uniform(1.0, 2.0, k)
    d4 = rng.uniform(-4.0, 4.0, k)
    x4 = d4 * rng.integers(-(1 << 20), 1 << 20, k).astype(np.float64)  # exact quotients (when d4*m is exact)
    # near midpoints: x = d * (q + 1/2 ulp) rounded, q random in [1, 2)
    q = rng.uniform(1.0, 2.0, k)
    d5 = rng.uniform(1.0, 2.0, k)
    x5 = d5 * (q + np.spacing(q) / 2)
    x6 = rng.integers(0, 2 ** 63, k, dtype=np.int64).view(np.float64)
    d6 = np.ones(k)  # divisor one, and powers of two below
    d6[::2] = 2.0 ** rng.integers(-1060, 1023, d6[::2].size).astype(np.float64)
    specials = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, 2.2250738585072014e-308, 1e-310,
                         1.7976931348623157e308, 2.0 ** 1021, 2.0 ** -960, 2.0 ** -959, 1.0, -3.0])
    xs, ds = np.meshgrid(specials, specials)
    x = np.concatenate([x1, x2, x3, x4, x5, x6, xs.ravel(), d1[:64], x2[:64] * 2.0 ** 600])
    d = np.concatenate([d1, d2, d3, d4, d5, d6, ds.ravel(), x1[:64], d2[:64] * 2.0 ** -900])
    return np.ascontiguousarray(x), np.ascontiguousarray(d)


def test_known_divisor_division_host_copy_is_ieee_division():
    x, d = division_pairs(1_200_000, 5)
    q = np.empty_like(x)
    bandlu.bandlu_selftest_div_host(x, d, q, x.size)
    with np.errstate(all="ignore"):
        ref = x / d
    bad = ~same_bits(q, ref)
    assert not bad.any(), list(zip(x[bad][:5], d[bad][:5]))


def test_quotient_with_zero_test_host_copy():
    """The back substitution's quotient (the CTA-wide solve): a zero dividend of either sign is
    kept as it is (the reference BLAS skips the division), which x / d would not do for a
    negative d; every other dividend is divided exactly as IEEE division does."""
    x, d = division_pairs(600_000, 23)
    x[:4000] = 0.0
    x[4000:8000] = -0.0
    d[:2000] = -np.abs(d[:2000])                      # +0 / negative and -0 / positive would flip
    d[6000:7000] = np.abs(d[6000:7000])
    q = np.empty_like(x)
    bandlu.bandlu_selftest_div_nz_host(x, d, q, x.size)
    with np.errstate(all="ignore"):
        ref = np.where(x != 0.0, x / d, x)
    bad = ~same_bits(q, ref)
    assert not bad.any(), list(zip(x[bad][:5], d[bad][:5]))
    assert np.signbit(q[:2000]).sum() == 0 and np.signbit(q[4000:8000]).all()


@pytest.mark.gpu
def test_known_divisor_division_device_is_ieee_division():
    import torch
    x, d = division_pairs(12_000_000, 17)
    xd = torch.from_numpy(x).cuda()
    dd = torch.from_numpy(d).cuda()
    q = torch.empty_like(xd)
    qd = torch.empty_like(xd)
    assert bandlu.bandlu_selftest_div_device(xd, dd, q, x.size, 0) == 0
    assert bandlu.bandlu_selftest_div_device(xd, dd, qd, x.size, 1) == 0
    torch.cuda.synchronize()
    q, qd = q.cpu().numpy(), qd.cpu().numpy()
    with np.errstate(all="ignore"):
        ref = x / d
    assert same_bits(q, qd).all(), list(zip(x[~same_bits(q, qd)][:5], d[~same_bits(q, qd)][:5]))
    assert same_bits(q, ref).all()
