"""Pins the oracle's routing simulator to what the paper and the mathematics
fix: hand-computed worked traces, the round-robin rule, least-loaded and the
length heuristic against an exhaustive scan re-derived from the outputs, the
one-instance pools where all policies coincide, closed forms for isolated
requests, the Pollaczek-Khinchine mean wait of the M/G/1 prefill queue,
learned-router limits that reduce to least-loaded, and conservation
invariants.  Capacity, budget and input errors are checked too."""
import numpy as np
import pytest

import simutil as U
from paper_2609_16206_gb300 import workloads as W


@pytest.mark.parametrize("case", U.worked_traces(), ids=lambda c: c["name"])
def test_worked_traces(orc, case):
    sc = U.sim_from(case["sim"])
    cc = U.consts_from(case["consts"])
    tr = U.trace_from(case["requests"])
    res = orc.simulate(sc, cc, case["policy"], tr)
    assert res["status"] == 0
    for key, val in case["expect"].items():
        if key in ("met", "p99_ttft_us"):
            continue
        assert res[key].tolist() == val, key
    if "met" in case["expect"]:
        met, p99 = orc.goodput(sc, tr, res["t_first_us"], res["t_done_us"])
        assert met == case["expect"]["met"]
        assert p99 == case["expect"]["p99_ttft_us"]


@pytest.fixture(scope="module")
def sweep_rows(orc):
    """A 2P+6D bursty replica and a 1P+3D Poisson replica under every policy."""
    out = []
    for wl, n in ((W.replica_sweep(), 3000), (W.single_replica(), 2000)):
        tr = orc.gen_trace(wl.trace, n, replica=1)
        for pol in W.ALL_POLICIES:
            res = orc.simulate(wl.sim, W.CALIBRATED, pol, tr)
            assert res["status"] == 0
            out.append((wl, pol, tr, res))
    return out


def test_round_robin_rule(sweep_rows):
    for wl, pol, tr, res in sweep_rows:
        if pol == W.POLICY_RR:
            k = np.arange(tr["arrival_us"].size)
            assert np.array_equal(res["i_pre"], k % wl.sim.n_prefill)
            assert np.array_equal(res["i_dec"], k % wl.sim.n_decode)


def test_least_loaded_is_exhaustive_argmin(sweep_rows):
    for wl, pol, tr, res in sweep_rows:
        if pol not in (W.POLICY_JSQ, W.POLICY_HEURISTIC):
            continue
        t = tr["arrival_us"]
        ip, idc = res["i_pre"].astype(np.int64), res["i_dec"].astype(np.int64)
        for k in range(t.size):
            qp = U.inflight_counts(t[k], ip, res["pre_end_us"], wl.sim.n_prefill, k)
            assert ip[k] == int(np.argmin(qp))
            if pol == W.POLICY_HEURISTIC and tr["pred_out"][k] >= wl.sim.heuristic_threshold_tokens:
                load = U.inflight_sums(t[k], idc, res["t_done_us"], tr["pred_out"], wl.sim.n_decode, k)
            else:
                load = U.inflight_counts(t[k], idc, res["t_done_us"], wl.sim.n_decode, k)
            assert idc[k] == int(np.argmin(load)), k


def test_learned_with_queue_weight_only_is_least_loaded(orc):
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2000, replica=4)
    qonly = W.CostConsts(w_b_q8=0, w_s_q8=0, w_q_us=5000)
    a = orc.simulate(wl.sim, qonly, W.POLICY_LEARNED, tr)
    b = orc.simulate(wl.sim, W.CALIBRATED, W.POLICY_JSQ, tr)
    for key in ("i_pre", "i_dec", "t_first_us", "t_done_us"):
        assert np.array_equal(a[key], b[key])


def test_learned_without_load_terms_picks_lowest_index(orc):
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 500, replica=2)
    flat = W.CostConsts(w_b_q8=0, w_q_us=0, rho_q8=0)
    res = orc.simulate(wl.sim, flat, W.POLICY_LEARNED, tr)
    assert not res["i_pre"].any() and not res["i_dec"].any()


def test_one_instance_pools_make_policies_identical(orc):
    sc = W.SimCfg(n_prefill=1, n_decode=1)
    tr = orc.gen_trace(W.TraceCfg(rate_mreq=(1500, 1500)), 1500)
    outs = [orc.simulate(sc, W.CALIBRATED, pol, tr) for pol in W.ALL_POLICIES]
    for o in outs[1:]:
        assert o["hash"] == outs[0]["hash"]
        assert np.array_equal(o["t_done_us"], outs[0]["t_done_us"])


def test_isolated_requests_closed_form(orc):
    rng = np.random.default_rng(5)
    n = 60
    p = rng.integers(16, 8193, n).astype(np.int32)
    o = rng.integers(1, 501, n).astype(np.int32)
    tr = {"arrival_us": (np.arange(n, dtype=np.int64) * 10_000_000), "prompt_len": p, "true_out": o,
          "pred_out": o.copy(), "slo_class": np.zeros(n, np.uint8)}
    sc = W.SimCfg(n_prefill=2, n_decode=3)
    for pol in W.ALL_POLICIES:
        res = orc.simulate(sc, W.CALIBRATED, pol, tr)
        assert res["status"] == 0
        for k in range(n):
            pk, ok = int(p[k]), int(o[k])
            ttft = 20_000 + 150 * pk + 20 * pk + 15_000 + 200 + pk // 1000
            tpot_sum = sum(15_000 + 200 + (pk + j) // 1000 for j in range(1, ok))
            assert res["t_first_us"][k] - tr["arrival_us"][k] == ttft
            assert res["t_done_us"][k] - res["t_first_us"][k] == tpot_sum


def test_prefill_queue_pollaczek_khinchine(orc):
    """M/G/1 FCFS prefill: mean wait = lambda E[S^2] / (2 (1 - lambda E[S]))."""
    rng = np.random.default_rng(21)
    n = 200_000
    p = rng.integers(16, 2001, n).astype(np.int32)
    lam = 1.0 / 0.36                         # req/s; E[S] = 20 ms + 0.15 ms * 1008 = 171.2 ms -> rho ~ 0.48
    gaps = np.floor(rng.exponential(1e6 / lam, n)).astype(np.int64)
    tr = {"arrival_us": np.cumsum(gaps), "prompt_len": p, "true_out": np.ones(n, np.int32),
          "pred_out": np.ones(n, np.int32), "slo_class": np.zeros(n, np.uint8)}
    sc = W.SimCfg(n_prefill=1, n_decode=1)
    res = orc.simulate(sc, W.CALIBRATED, W.POLICY_RR, tr)
    assert res["status"] == 0
    s = (20_000 + 150 * p.astype(np.float64)) / 1e6
    wait = (res["pre_end_us"] - tr["arrival_us"]) / 1e6 - s
    assert wait.min() >= 0
    lam_hat = n / (tr["arrival_us"][-1] / 1e6)
    pk = lam_hat * np.mean(s * s) / (2 * (1 - lam_hat * np.mean(s)))
    assert abs(wait.mean() / pk - 1) < 0.08


def test_conservation_invariants(sweep_rows):
    for wl, pol, tr, res in sweep_rows:
        sc = wl.sim
        a, p, o = tr["arrival_us"], tr["prompt_len"].astype(np.int64), tr["true_out"].astype(np.int64)
        assert np.all(res["pre_end_us"] >= a + sc.pre_base_us + sc.pre_us_per_tok * p)
        assert np.array_equal(res["t_ready_us"], res["pre_end_us"] + sc.xfer_us_per_tok * p)
        assert np.all(res["t_first_us"] > res["t_ready_us"])
        assert np.all(res["t_done_us"] >= res["t_first_us"] + (o - 1) * sc.dec_base_us)
        assert res["stats"]["max_reserved"] <= sc.kv_cap_tokens
        # every request is active at least over [t_first, t_done]: reservations then fit
        for d in range(sc.n_decode):
            on = res["i_dec"] == d
            for t in np.unique(res["t_first_us"][on])[::37]:
                act = on & (res["t_first_us"] <= t) & (res["t_done_us"] >= t)
                assert (p[act] + o[act]).sum() <= sc.kv_cap_tokens
        # prefill FCFS: per instance, in arrival order, ends strictly increase
        for i in range(sc.n_prefill):
            e = res["pre_end_us"][res["i_pre"] == i]
            assert np.all(np.diff(e) > 0)
        # total decode steps cover every generated token at least once per step
        assert res["stats"]["steps"] * 1 >= o.max()


def test_hash_matches_outputs(orc, sweep_rows):
    for wl, pol, tr, res in sweep_rows[:2]:
        h = orc.row_hash(res["i_pre"], res["i_dec"], res["t_first_us"], res["t_done_us"])
        assert h == res["hash"]
        t2 = res["t_done_us"].copy()
        t2[17] += 1
        assert orc.row_hash(res["i_pre"], res["i_dec"], res["t_first_us"], t2) != h


def test_capacity_overflow_exact(orc):
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2000, replica=0)
    base = orc.simulate(wl.sim, W.CALIBRATED, W.POLICY_LEARNED, tr)
    st = base["stats"]
    caps = dict(cap_pending=st["max_pending"], cap_waiting=st["max_waiting"], cap_active=st["max_active"],
                cap_prefill_ring=st["max_prefill"])
    ok = orc.simulate(wl.sim.replace(**caps), W.CALIBRATED, W.POLICY_LEARNED, tr)
    assert ok["status"] == 0 and ok["hash"] == base["hash"]
    for name in caps:
        tight = dict(caps)
        tight[name] -= 1
        if tight[name] < 1:
            continue
        bad = orc.simulate(wl.sim.replace(**tight), W.CALIBRATED, W.POLICY_LEARNED, tr)
        assert bad["status"] == orc.EOVERFLOW, name


def test_step_budget_timeout(orc):
    wl = W.single_replica()
    tr = orc.gen_trace(wl.trace, 300)
    res = orc.simulate(wl.sim.replace(max_steps_per_instance=50), W.CALIBRATED, W.POLICY_RR, tr)
    assert res["status"] == orc.ETIMEOUT


@pytest.mark.parametrize("field,value", [("prompt_len", -1), ("true_out", 0), ("pred_out", -3),
                                         ("slo_class", 2), ("arrival_us", -5)])
def test_invalid_request_rejected(orc, field, value):
    wl = W.single_replica()
    tr = orc.gen_trace(wl.trace, 50)
    tr[field] = tr[field].copy()
    tr[field][10] = value
    assert orc.simulate(wl.sim, W.CALIBRATED, W.POLICY_LEARNED, tr)["status"] == orc.EINVAL


def test_unsorted_arrivals_and_oversized_request_rejected(orc):
    wl = W.single_replica()
    tr = orc.gen_trace(wl.trace, 50)
    t = dict(tr)
    t["arrival_us"] = tr["arrival_us"].copy()
    t["arrival_us"][20] = t["arrival_us"][19] - 1
    assert orc.simulate(wl.sim, W.CALIBRATED, 0, t)["status"] == orc.EINVAL
    small = wl.sim.replace(kv_cap_tokens=int(tr["prompt_len"].max()))
    assert orc.simulate(small, W.CALIBRATED, 0, tr)["status"] == orc.EINVAL


def test_empty_trace(orc):
    wl = W.single_replica()
    tr = orc.gen_trace(wl.trace, 0)
    res = orc.simulate(wl.sim, W.CALIBRATED, 0, tr)
    assert res["status"] == 0 and res["hash"] == 0
