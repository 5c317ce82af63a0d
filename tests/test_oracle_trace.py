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


def test_mmpp_starts_in_the_low_state(orc):
    """The two-state MMPP starts in its first (low-rate) state: over many
    replicas the arrivals in the first second average about 3 (the first
    dwell, mean 10 s, rarely ends that early: e^-0.1 of replicas are still in
    it at 1 s), not 12; listing the rates the other way round flips it.  The
    mean rate and the dispersion test above cannot tell which state comes
    first."""
    tc = W.replica_sweep().trace
    n_rep = 2000

    def first_second_mean(cfg):
        counts = [int(np.sum(orc.gen_trace(cfg, 40, replica=g)["arrival_us"] < 1_000_000)) for g in range(n_rep)]
        return float(np.mean(counts))

    # exact expectation: rate lam0 until the first switch (exponential, mean 10 s), then lam1
    # E[count in [0, 1 s)] = lam1 * 1 + (lam0 - lam1) * E[min(D, 1)], E[min(D, 1)] = 10 (1 - e^-0.1)
    e_min = 10.0 * (1.0 - np.exp(-0.1))
    low_first = 12.0 + (3.0 - 12.0) * e_min
    high_first = 3.0 + (12.0 - 3.0) * e_min
    se = np.sqrt(12.0 / n_rep)
    a = first_second_mean(tc)
    b = first_second_mean(tc.replace(rate_mreq=(tc.rate_mreq[1], tc.rate_mreq[0])))
    assert abs(a - low_first) < 5 * se, (a, low_first)
    assert abs(b - high_first) < 5 * se, (b, high_first)


def test_counter_layout_of_each_request(orc):
    """The trace spec's counter layout, checked against the KAT-pinned
    Philox4x32-10 and the separately pinned fp32 functions: replica g uses key
    seed + (g mod n_seeds) and sub-stream g / n_seeds; request k draws counter
    (k, sub, 0, 0) for (prompt, mixture, output, noise) and (k, sub, 0, 1) for
    (class, gap); MMPP dwell j draws (j, sub, 1, 0).  Every field of a few
    requests of several replicas is rebuilt here from those words."""
    tc = W.TraceCfg(seed=11, n_seeds=3, arrival_kind=0, rate_mreq=(4000, 4000))
    f32 = np.float32

    def round_clip(v, lo, hi):
        y = f32(v) + f32(0.5)
        if not (y < f32(hi)):
            return hi
        return max(lo, int(y))

    for g in (0, 1, 2, 4, 7):
        tr = orc.gen_trace(tc, 40, replica=g)
        seed = tc.seed + g % tc.n_seeds
        key = [seed & 0xFFFFFFFF, seed >> 32]
        sub = g // tc.n_seeds
        lam = 0
        for k in range(40):
            x = orc.philox4x32_10([k, sub, 0, 0], key)
            y = orc.philox4x32_10([k, sub, 0, 1], key)
            zp = orc.det_ndtrif(np.array([x[0]], np.uint32))[0]
            p = round_clip(orc.det_expf(np.array([f32(tc.prompt_mu) + f32(tc.prompt_sigma) * zp], f32))[0],
                           tc.prompt_min, tc.prompt_max)
            short = int(x[1]) < tc.mix_short_thr
            mu, sg = (tc.short_mu, tc.short_sigma) if short else (tc.long_mu, tc.long_sigma)
            zo = orc.det_ndtrif(np.array([x[2]], np.uint32))[0]
            o = round_clip(orc.det_expf(np.array([f32(mu) + f32(sg) * zo], f32))[0], tc.out_min, tc.out_max)
            zn = orc.det_ndtrif(np.array([x[3]], np.uint32))[0]
            fac = orc.det_expf(np.array([f32(tc.noise_sigma) * zn], f32))[0]
            oh = round_clip(f32(o) * fac, tc.pred_min, tc.pred_max)
            c = int(int(y[0]) >= tc.class_thr[0])
            lg = orc.det_logf(orc.unit_uniform(np.array([y[1]], np.uint32)))[0]
            lam += int(f32(-lg) * f32(1e9))
            assert (int(tr["prompt_len"][k]), int(tr["true_out"][k]), int(tr["pred_out"][k]),
                    int(tr["slo_class"][k])) == (p, o, oh, c), (g, k)
            assert int(tr["arrival_us"][k]) == lam // tc.rate_mreq[0], (g, k)

    # MMPP: the first dwell comes from counter (0, sub, 1, 0) of the replica's key
    mm = W.TraceCfg(seed=5, arrival_kind=1, rate_mreq=(3000, 12000), dwell_mean_us=10_000_000)
    tr = orc.gen_trace(mm, 400, replica=0)
    w = orc.philox4x32_10([0, 0, 1, 0], [5, 0])
    d0 = int(f32(-orc.det_logf(orc.unit_uniform(np.array([w[0]], np.uint32)))[0]) * f32(mm.dwell_mean_us))
    # arrivals before the first switch follow the low rate exactly
    lam = 0
    for k in range(400):
        y = orc.philox4x32_10([k, 0, 0, 1], [5, 0])
        lam += int(f32(-orc.det_logf(orc.unit_uniform(np.array([y[1]], np.uint32)))[0]) * f32(1e9))
        if lam >= 3000 * d0:
            break
        assert int(tr["arrival_us"][k]) == lam // 3000, k
    assert k > 0
