"""Parity of the sweep workloads built on the saturation search: the
bisection's endpoints re-checked by the oracle, the mispriced-constants x
pool-width sweep and the scarcity stress on a large pool (reduced, and at the
full workload sizes with sampled rows compared by hash)."""
import numpy as np
import pytest
import torch

from gpuutil import host_trace, need_gpu
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _oracle_rr_goodput(orc, tc, sc, rate, n_req):
    law = tc.replace(arrival_kind=0, rate_mreq=(rate, rate))
    tr = orc.gen_trace(law, n_req, replica=0)
    res = orc.simulate(sc, W.CALIBRATED, W.POLICY_RR, tr)
    if res["status"] != 0:
        return None
    return orc.goodput(sc, tr, res["t_first_us"], res["t_done_us"])[0]


def test_saturation_bisection_endpoints(orc):
    need_gpu()
    from paper_2609_16206_gb300 import sweep
    sc = W.SimCfg(n_prefill=2, n_decode=3)
    laws = [W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(m)) for m in (1.0, 0.5)]
    n, lo0, hi0 = 2000, 1, 40_000
    rates = sweep.saturation_rate(laws, sc, n_req=n, lo=lo0, hi=hi0, steps=16)
    for law, r in zip(laws, rates):
        assert lo0 < r < hi0
        assert 2 * _oracle_rr_goodput(orc, law, sc, r, n) >= n
        above = _oracle_rr_goodput(orc, law, sc, r + 1, n)
        assert above is None or 2 * above < n


def _run_sets(ctr, sc, sets, pols, tr, R, N):
    rows = R * len(sets) * len(pols)
    tf = torch.empty((rows, N), dtype=torch.int64, device="cuda")
    td = torch.empty_like(tf)
    h = torch.empty(rows, dtype=torch.int64, device="cuda")
    st = torch.empty(rows, dtype=torch.int32, device="cuda")
    ws = ctr.simulate_workspace(sc, rows, N, "cuda")
    ctr.ctr_simulate(sc, sets, pols, tr, R, N, tf, td, h, st, ws)
    torch.cuda.synchronize()
    return h.cpu().numpy().astype(np.uint64), st.cpu().numpy()


def _calibration_case(orc, widths, mixes, loads, seeds, n_req, n_bisect, sample):
    ctr = need_gpu()
    from paper_2609_16206_gb300 import sweep
    sets = W.mispriced_sets()
    checked = 0
    for w in widths:
        sc = W.SimCfg(n_prefill=2, n_decode=w)
        laws = [W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(m)) for m in mixes]
        sat = sweep.saturation_rate(laws, sc, n_req=n_bisect)
        for law, s_rate in zip(laws, sat):
            for load in loads:
                rate = sweep.load_rate(s_rate, load)
                tc = law.replace(rate_mreq=(rate, rate))
                tr = ctr.empty_requests(seeds, n_req, "cuda")
                ctr.ctr_gen_trace(tc, seeds, 0, n_req, tr)
                h_l, st_l = _run_sets(ctr, sc, sets, [W.POLICY_LEARNED], tr, seeds, n_req)
                h_b, st_b = _run_sets(ctr, sc, [W.CALIBRATED], [1, 2, 3], tr, seeds, n_req)
                assert (st_l == 0).all() or (st_l[st_l != 0] == ctr.CTR_EOVERFLOW).all()
                for r in sample(seeds):
                    trh = host_trace(tr, r)
                    for si in (0, 1, 64):
                        o = orc.simulate(sc, sets[si], W.POLICY_LEARNED, trh)
                        assert st_l[r * len(sets) + si] == o["status"]
                        if o["status"] == 0:
                            assert int(h_l[r * len(sets) + si]) == o["hash"]
                        checked += 1
                    for j, pol in enumerate((1, 2, 3)):
                        o = orc.simulate(sc, W.CALIBRATED, pol, trh)
                        assert st_b[r * 3 + j] == o["status"]
                        if o["status"] == 0:
                            assert int(h_b[r * 3 + j]) == o["hash"]
    return checked


def test_calibration_sweep_reduced(orc):
    assert _calibration_case(orc, widths=(4, 7), mixes=(1.0, 0.5), loads=(0.8, 1.3), seeds=2, n_req=1500,
                             n_bisect=1500, sample=lambda s: range(s)) > 0


def test_calibration_sweep_full_size_sampled(orc):
    """5 widths x 4 mixes x 4 loads x 16 seeds x (65 learned sets + 3 baselines), 10,000 requests;
    every row's status checked, rows sampled against the oracle by hash."""
    assert _calibration_case(orc, widths=(3, 4, 5, 6, 7), mixes=(1.0, 5 / 6, 2 / 3, 0.5),
                             loads=(0.8, 29 / 30, 17 / 15, 1.3), seeds=16, n_req=10_000, n_bisect=10_000,
                             sample=lambda s: (0,)) > 0


def _large_pool_case(orc, n_replicas, n_req, sample_replicas):
    ctr = need_gpu()
    from paper_2609_16206_gb300 import sweep
    base = W.large_pool()
    sat = sweep.saturation_rate([base.trace], base.sim, n_req=10_000)[0]
    rate = sweep.load_rate(sat, 1.2)
    tc = base.trace.replace(rate_mreq=(rate, rate))
    tr = ctr.empty_requests(n_replicas, n_req, "cuda")
    ctr.ctr_gen_trace(tc, n_replicas, 0, n_req, tr)
    h, st = _run_sets(ctr, base.sim, base.consts, list(W.ALL_POLICIES), tr, n_replicas, n_req)
    assert (st == 0).all(), np.unique(st)
    for r in sample_replicas:
        trh = host_trace(tr, r)
        for j, pol in enumerate(W.ALL_POLICIES):
            o = orc.simulate(base.sim, base.consts[0], pol, trh)
            assert o["status"] == 0 and int(h[r * 4 + j]) == o["hash"], (r, pol)
    return sat


def test_large_pool_stress_reduced(orc):
    sat = _large_pool_case(orc, n_replicas=8, n_req=5000, sample_replicas=(0, 7))
    assert sat > 1000


def test_large_pool_stress_full_size_sampled(orc):
    """16,384 replicas x 50,000 requests, 4P+28D at 1.2x the saturation rate, all four policies."""
    _large_pool_case(orc, n_replicas=16384, n_req=50_000, sample_replicas=(0, 16383))


def test_noise_sweep(orc):
    """sec. V-G: predictor noise 0..150 % on the same replicas, one launch; sampled rows = oracle, and the
    learned router's routes depend on the noise while round-robin's do not."""
    ctr = need_gpu()
    from paper_2609_16206_gb300 import sweep
    wl = W.replica_sweep(n_req=2000)
    seeds = 3
    buf, R = sweep.noise_sweep(wl, seeds=seeds)
    torch.cuda.synchronize()
    h = buf.row_hash.cpu().numpy().astype(np.uint64)
    st = buf.row_status.cpu().numpy()
    assert (st == 0).all()
    n_pol = len(W.ALL_POLICIES)
    for i, sg in enumerate(sweep.NOISE_SIGMAS):
        r = i * seeds + 1
        trh = host_trace(buf.trace, r)
        ref = orc.gen_trace(wl.trace.replace(noise_sigma=sg), wl.n_req, replica=1)
        for key in ref:
            assert np.array_equal(trh[key], ref[key]), key
        for j, pol in enumerate(W.ALL_POLICIES):
            assert int(h[r * n_pol + j]) == orc.simulate(wl.sim, W.CALIBRATED, pol, trh)["hash"]
    rr = [int(h[(i * seeds) * n_pol + 1]) for i in range(len(sweep.NOISE_SIGMAS))]
    lr = [int(h[(i * seeds) * n_pol + 0]) for i in range(len(sweep.NOISE_SIGMAS))]
    assert len(set(rr)) == 1 and len(set(lr)) == len(lr)


def test_calibration_sweep_batched(orc):
    """The batched calibration sweep: one trace buffer and two launches per width; sampled rows = oracle."""
    ctr = need_gpu()
    from paper_2609_16206_gb300 import sweep
    widths, mixes, loads, seeds, n = (3, 6), (1.0, 0.5), (0.8, 1.3), 2, 1500
    sat = sweep.calibration_saturation(widths, mixes, n_req=n)
    out = sweep.calibration_sweep(sat, widths, mixes, loads, seeds, n_req=n)
    torch.cuda.synchronize()
    sets = W.mispriced_sets()
    for w, (lb, bb) in out.items():
        sc = W.SimCfg(n_prefill=2, n_decode=w)
        st_l = lb.row_status.cpu().numpy()
        h_l = lb.row_hash.cpu().numpy().astype(np.uint64)
        st_b = bb.row_status.cpu().numpy()
        h_b = bb.row_hash.cpu().numpy().astype(np.uint64)
        for i, mix in enumerate(mixes):
            for j, load in enumerate(loads):
                r = (i * len(loads) + j) * seeds + (i + j) % seeds
                trh = host_trace(lb.trace, r)
                rate = sweep.load_rate(sat[w][i], load)
                ref = orc.gen_trace(W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(mix), rate_mreq=(rate, rate)),
                                    n, replica=(i + j) % seeds)
                assert np.array_equal(trh["arrival_us"], ref["arrival_us"])
                for si in (0, 21, 64):
                    o = orc.simulate(sc, sets[si], W.POLICY_LEARNED, trh)
                    assert st_l[r * len(sets) + si] == o["status"]
                    if o["status"] == 0:
                        assert int(h_l[r * len(sets) + si]) == o["hash"]
                for b, pol in enumerate((W.POLICY_RR, W.POLICY_JSQ, W.POLICY_HEURISTIC)):
                    o = orc.simulate(sc, W.CALIBRATED, pol, trh)
                    assert st_b[r * 3 + b] == o["status"]
                    if o["status"] == 0:
                        assert int(h_b[r * 3 + b]) == o["hash"]


def test_policy_table_is_the_mean_of_oracle_rows(orc):
    """Table 2's columns per policy: the mean over replicas of each row's goodput, P99 TTFT and P99 TPOT,
    every row recomputed by the oracle from the oracle's own simulation of the same trace."""
    from paper_2609_16206_gb300 import ctr, sweep
    need_gpu()
    wl = W.replica_sweep(n_replicas=3, n_req=3000)
    table = sweep.policy_table(wl)
    tr = ctr.empty_requests(wl.n_replicas, wl.n_req, "cuda")
    ctr.ctr_gen_trace(wl.trace, wl.n_replicas, 0, wl.n_req, tr)
    torch.cuda.synchronize()
    for pol in wl.policies:
        gp, ttft, tpot = [], [], []
        for r in range(wl.n_replicas):
            trh = host_trace(tr, r)
            o = orc.simulate(wl.sim, wl.consts[0], pol, trh)
            met, p99 = orc.goodput(wl.sim, trh, o["t_first_us"], o["t_done_us"])
            gp.append(met / wl.n_req)
            ttft.append(p99 / 1e6)
            tpot.append(orc.p99_tpot(trh, o["t_first_us"], o["t_done_us"]) / 1e6)
        row = table[W.POLICY_NAMES[pol]]
        assert row["rows_failed"] == 0
        assert row["goodput"] == pytest.approx(np.mean(gp), rel=1e-12)
        assert row["p99_ttft_s"] == pytest.approx(np.mean(ttft), rel=1e-12)
        assert row["p99_tpot_s"] == pytest.approx(np.mean(tpot), rel=1e-12)


def test_resumable_sweep_equals_one_shot(orc, tmp_path):
    """A sweep stopped after its first chunk and resumed from its journal gives, row for row, the
    checksums, statuses, met counts and P99 TTFTs of one launch over all replicas (chunks of 3, 3 and 1
    replicas from their own trace offsets)."""
    from paper_2609_16206_gb300 import ctr, sweep
    need_gpu()
    wl = W.replica_sweep(n_replicas=7, n_req=1500)
    j = str(tmp_path / "journal")
    assert sweep.resumable_sweep(wl, j, chunk=3, max_chunks=1) is None
    res = sweep.resumable_sweep(wl, j, chunk=3)
    rows = wl.n_replicas * len(wl.policies)
    buf = sweep.alloc(wl.sim, wl.n_replicas, rows, wl.n_req, "cuda")
    sweep.run_step(wl.trace, wl.sim, wl.consts, list(wl.policies), wl.n_replicas, wl.n_req, 0, buf)
    torch.cuda.synchronize()
    assert np.array_equal(res["row_hash"], buf.row_hash.cpu().numpy().astype(np.uint64))
    assert np.array_equal(res["row_status"], buf.row_status.cpu().numpy())
    assert np.array_equal(res["met"], buf.met.cpu().numpy())
    assert np.array_equal(res["p99_ttft_us"], buf.p99.cpu().numpy())
    assert (res["row_status"] == ctr.CTR_OK).all()
    trh = host_trace(buf.trace, 6)  # the last chunk's replica against the oracle
    for j_, pol in enumerate(wl.policies):
        assert int(res["row_hash"][6 * len(wl.policies) + j_]) == orc.simulate(wl.sim, wl.consts[0], pol, trh)["hash"]
