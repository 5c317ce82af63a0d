"""Pins the oracle's deterministic fp32 log / exp / normal quantile (the
precision the trace's integer decisions are defined in) against the host's
fp64 libm / scipy, and exact special values."""
import numpy as np
import scipy.special as sp


def _ulps32(got, ref64):
    """error of fp32 results in units of the fp32 spacing at the exact value"""
    return np.max(np.abs(got.astype(np.float64) - ref64) / np.spacing(np.abs(ref64).astype(np.float32)))


def test_logf_against_libm(orc):
    rng = np.random.default_rng(11)
    x = np.concatenate([rng.random(50_000), 10.0 ** rng.uniform(-37, 38, 50_000),
                        orc.unit_uniform(rng.integers(0, 2**32, 50_000, dtype=np.uint64))]).astype(np.float32)
    x = x[x > 0]
    ref = np.log(x.astype(np.float64))
    big = np.abs(ref) > 1e-3           # away from the zero of log, where ulps are relative to a tiny value
    assert _ulps32(orc.det_logf(x)[big], ref[big]) <= 3.0
    small = ~big
    assert np.max(np.abs(orc.det_logf(x)[small] - ref[small]) / np.abs(ref[small] + 1e-30)) < 1e-6


def test_logf_special_values(orc):
    v = orc.det_logf(np.array([1.0, 2.0, 0.5], np.float32))
    assert v[0] == 0.0 and v[1] == -v[2]
    assert abs(v[1] - np.log(2.0)) <= np.spacing(np.float32(np.log(2.0)))


def test_expf_against_libm(orc):
    rng = np.random.default_rng(12)
    x = np.concatenate([rng.uniform(-87, 88, 50_000), rng.uniform(-12, 12, 50_000)]).astype(np.float32)
    assert _ulps32(orc.det_expf(x), np.exp(x.astype(np.float64))) <= 2.0
    e = orc.det_expf(np.array([0.0, -0.0, 1.0], np.float32))
    assert e[0] == 1.0 and e[1] == 1.0
    assert abs(e[2] - np.e) <= np.spacing(np.float32(np.e))


def test_unit_uniform_is_one_rounding(orc):
    rng = np.random.default_rng(14)
    u = rng.integers(0, 2**32, 100_000, dtype=np.uint64)
    exact = (u.astype(np.float64) + 0.5) * 2.0**-32
    got = orc.unit_uniform(u)
    assert np.array_equal(got, exact.astype(np.float32))        # numpy's rounding of the exact value
    comp = orc.unit_uniform(~u.astype(np.uint32))
    assert np.array_equal(comp, (1.0 - exact).astype(np.float32))


def test_ndtrif_against_scipy(orc):
    rng = np.random.default_rng(13)
    u = np.concatenate([rng.integers(0, 2**32, 200_000, dtype=np.uint64),
                        np.array([0, 1, 2**31 - 1, 2**31, 2**32 - 1, 2**32 - 2], np.uint64)])
    U = (u.astype(np.float64) + 0.5) * 2.0**-32
    ref = sp.ndtri(U)
    got = orc.det_ndtrif(u).astype(np.float64)
    assert np.max(np.abs(got - ref) / np.maximum(np.abs(ref), 0.05)) < 2e-6


def test_ndtrif_symmetry_and_cdf(orc):
    u = np.arange(0, 2**32, 2**16 + 1, dtype=np.uint64)
    a = orc.det_ndtrif(u)
    b = orc.det_ndtrif((~u.astype(np.uint32)).astype(np.uint64))
    assert np.array_equal(a, -b)                                   # exact antisymmetry by construction
    U = (u.astype(np.float64) + 0.5) * 2.0**-32
    assert np.max(np.abs(sp.ndtr(a.astype(np.float64)) - U)) < 2e-7
