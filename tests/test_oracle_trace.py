"""Pins the oracle's synthetic trace: exact discretised lognormal moments,
class and mixture proportions, Poisson gaps (KS), MMPP mean rate and index of
dispersion (closed form of the two-state MMPP), and the replica seeding rule."""
import numpy as np
import pytest
from scipy import stats

from paper_2609_16206_gb300 import workloads as W

N = 200_000


@pytest.fixture(scope="module")
def trace(orc):
    return orc.gen_trace(W.TraceCfg(), N)


def _rounded_lognormal_pmf(mu, sigma, lo, hi):
    """P(clip(floor(X + 1/2), lo, hi) = v) for X ~ LN(mu, sigma), v = lo..hi."""
    d = stats.lognorm(s=sigma, scale=np.exp(mu))
    v = np.arange(lo, hi + 1, dtype=np.float64)
    cdf_hi = d.cdf(v + 0.5)
    cdf_lo = d.cdf(v - 0.5)
    pmf = cdf_hi - cdf_lo
    pmf[0] = d.cdf(lo + 0.5)
    pmf[-1] = d.sf(hi - 0.5)
    return v, pmf


def _check_mean(sample, v, pmf):
    mean = float(np.sum(v * pmf))
    var = float(np.sum(v * v * pmf)) - mean * mean
    se = np.sqrt(var / sample.size)
    assert abs(sample.mean() - mean) < 4.5 * se, (sample.mean(), mean, se)
    return mean


def test_prompt_length_law(trace):
    p = trace["prompt_len"]
    assert p.min() >= 16 and p.max() <= 8192
    v, pmf = _rounded_lognormal_pmf(W.LN_512, 1.0, 16, 8192)
    mean = _check_mean(p, v, pmf)
    assert 830 < mean < 840
    # chi-square over 20 equiprobable-ish bins of the exact pmf
    edges = np.searchsorted(np.cumsum(pmf), np.linspace(0, 1, 21)[1:-1])
    obs = np.bincount(np.searchsorted(v[edges], p, side="left"), minlength=20)
    exp = np.array([pmf[a:b].sum() for a, b in zip(np.r_[0, edges], np.r_[edges, v.size])]) * p.size
    chi2 = np.sum((obs - exp) ** 2 / exp)
    assert stats.chi2.sf(chi2, df=19) > 1e-4


def test_output_length_mixture(trace):
    o = trace["true_out"]
    assert o.min() >= 1 and o.max() <= 4096
    v, pmf_s = _rounded_lognormal_pmf(W.LN_128, 0.8, 1, 4096)
    _, pmf_l = _rounded_lognormal_pmf(W.LN_1024, 0.6, 1, 4096)
    _check_mean(o, v, 0.7 * pmf_s + 0.3 * pmf_l)


def test_predicted_length_noise(trace):
    o = trace["true_out"].astype(np.float64)
    oh = trace["pred_out"].astype(np.float64)
    big = o >= 1000
    r = np.log(oh[big] / o[big])
    assert abs(r.mean()) < 0.01
    assert abs(r.std() - 0.3) < 0.01


def test_no_noise_means_exact_prediction(orc):
    tr = orc.gen_trace(W.TraceCfg(noise_sigma=0.0), 5000)
    assert np.array_equal(tr["pred_out"], tr["true_out"])


def test_class_proportions(orc, trace):
    c = trace["slo_class"]
    assert set(np.unique(c)) == {0, 1}
    assert abs((c == 0).mean() - 0.6) < 4.5 * np.sqrt(0.24 / N)
    tc3 = W.large_pool().trace
    c3 = orc.gen_trace(tc3, N)["slo_class"]
    for cls, prob in enumerate((0.3, 0.4, 0.3)):
        assert abs((c3 == cls).mean() - prob) < 4.5 * np.sqrt(prob * (1 - prob) / N)


def test_poisson_gaps_exponential(trace):
    t = trace["arrival_us"]
    assert np.all(np.diff(t) >= 0)
    gaps = np.diff(np.r_[0, t]).astype(np.float64)
    mean_us = 1e6 / 4.0
    assert abs(gaps.mean() / mean_us - 1) < 4.5 / np.sqrt(N)
    ks = stats.kstest(gaps + 0.5, stats.expon(scale=mean_us).cdf)
    assert ks.pvalue > 1e-4


def test_mmpp_rate_and_dispersion(orc):
    tc = W.replica_sweep().trace
    t = orc.gen_trace(tc, N)["arrival_us"]
    assert np.all(np.diff(t) >= 0)
    span_s = t[-1] / 1e6
    assert abs(N / span_s - 7.5) < 0.4          # (3 + 12) / 2 with equal mean dwell
    w = 100.0                                   # window, s
    counts = np.bincount((t / 1e6 // w).astype(np.int64))[:-1]
    idx = counts.var() / counts.mean()
    r = 2 * 0.1                                 # switching rate sum (1 / 10 s each way)
    lam0, lam1, lbar = 3.0, 12.0, 7.5
    closed = 1 + 2 * (lam1 - lam0) ** 2 * 0.25 / (lbar * r * r * w) * (r * w - 1 + np.exp(-r * w))
    assert 0.65 * closed < idx < 1.35 * closed


def test_replica_seeding_rule(orc):
    tc = W.TraceCfg(seed=7, n_seeds=3, arrival_kind=1, rate_mreq=(3000, 12000))
    for g in (0, 1, 2, 5, 11):
        a = orc.gen_trace(tc, 300, replica=g)
        b = orc.gen_trace(tc.replace(seed=7 + g % 3, n_seeds=1), 300, replica=g // 3)
        for key in a:
            assert np.array_equal(a[key], b[key])
    r0 = orc.gen_trace(tc, 300, replica=0)
    r3 = orc.gen_trace(tc, 300, replica=3)
    assert not np.array_equal(r0["prompt_len"], r3["prompt_len"])
    again = orc.gen_trace(tc, 300, replica=0)
    assert all(np.array_equal(r0[k], again[k]) for k in r0)
