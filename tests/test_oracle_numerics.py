"""Pins the oracle's deterministic fp64 log / exp / normal quantile against the
host's libm / scipy (a few ulp) and exact special values."""
import numpy as np
import pytest
import scipy.special as sp


def _ulps(a, b):
    return np.max(np.abs(a - b) / np.spacing(np.abs(b)))


def test_log_against_libm(orc):
    rng = np.random.default_rng(11)
    x = np.concatenate([rng.random(50_000), 10.0 ** rng.uniform(-300, 300, 50_000),
                        (rng.integers(0, 2**32, 50_000) + 0.5) * 2.0**-32])
    assert _ulps(orc.det_log(x), np.log(x)) <= 3.0


def test_log_special_values(orc):
    assert orc.det_log(np.array([1.0]))[0] == 0.0
    two = orc.det_log(np.array([2.0, 0.5, 1024.0]))
    assert abs(two[0] - np.log(2.0)) <= np.spacing(np.log(2.0))
    assert two[1] == -two[0]
    assert abs(two[2] - 10 * np.log(2.0)) <= 2 * np.spacing(10 * np.log(2.0))


def test_exp_against_libm(orc):
    rng = np.random.default_rng(12)
    x = np.concatenate([rng.uniform(-700, 700, 50_000), rng.uniform(-30, 30, 50_000)])
    assert _ulps(orc.det_exp(x), np.exp(x)) <= 2.0
    e = orc.det_exp(np.array([0.0, -0.0, 1.0]))
    assert e[0] == 1.0 and e[1] == 1.0
    assert abs(e[2] - np.e) <= np.spacing(np.e)


def test_exp_log_roundtrip(orc):
    x = np.linspace(0.01, 50.0, 5001)
    assert np.max(np.abs(orc.det_exp(orc.det_log(x)) / x - 1.0)) < 1e-14


def test_ndtri_against_scipy(orc):
    rng = np.random.default_rng(13)
    u = np.concatenate([(rng.integers(0, 2**32, 100_000) + 0.5) * 2.0**-32, 10.0 ** rng.uniform(-300, -2, 5000),
                        np.array([0.075, 0.925, 0.5 - 1e-9, 1e-300])])
    ref = sp.ndtri(u)
    got = orc.det_ndtri(u)
    assert np.max(np.abs(got - ref) / np.maximum(np.abs(ref), 1e-300)) < 5e-15


def test_ndtri_symmetry_and_centre(orc):
    u = (np.arange(1, 2**16) + 0.5) * 2.0**-16
    a = orc.det_ndtri(u)
    b = orc.det_ndtri(1.0 - u)
    assert np.max(np.abs(a + b)) < 1e-14
    assert orc.det_ndtri(np.array([0.5]))[0] == 0.0
    # the normal CDF recovers the probability
    assert np.max(np.abs(sp.ndtr(a) - u)) < 1e-14
