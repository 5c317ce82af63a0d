"""Pins for the router signals of the deployed proxy (sec. IV-A, discussed in
sec. VI): backlog from an in-flight ledger priced with the router's own
constants, and KV occupancy polled on a fixed period.  Each oracle mode is
checked against a re-derivation from its own outputs, against modes it must
reduce to, and against the unit argument of sec. III-B."""
import numpy as np
import pytest

from paper_2609_16206_gb300 import workloads as W

B_CLAMP = 1 << 40


def _rederive(tr, res, sc, cc):
    """Replay every routing decision of a learned row whose pressure feature is
    ablated, from the row's outputs: the prefill ledger holds the requests
    whose prefill has not ended at t_k, the decode ledger those not completed
    at t_k; each is priced once with the router's constants."""
    t = tr["arrival_us"].astype(np.int64)
    p = tr["prompt_len"].astype(np.int64)
    oh = tr["pred_out"].astype(np.int64)
    cls = tr["slo_class"].astype(np.int64)
    ip, idc = res["i_pre"].astype(np.int64), res["i_dec"].astype(np.int64)
    pre_end, done = res["pre_end_us"], res["t_done_us"]
    work_pre = cc.tau_pre0_us + cc.tau_pre_us * p
    work_dec = oh * cc.tau_dec_us
    for k in range(t.size):
        tk = int(t[k])
        sig = int(cc.sigma_q8[cls[k]])
        best = None
        for i in range(sc.n_prefill):
            m = (ip[:k] == i) & (pre_end[:k] > tk)
            led = min(B_CLAMP, int(work_pre[:k][m].sum()))
            cost = (cc.w_b_q8 * led + cc.w_s_q8 * int(work_pre[k])) * sig + cc.w_q_us * int(m.sum()) * 65536
            if best is None or cost < best[0]:
                best = (cost, i)
        assert best[1] == ip[k], k
        best = None
        for d in range(sc.n_decode):
            m = (idc[:k] == d) & (done[:k] > tk)
            led = min(B_CLAMP, int(work_dec[:k][m].sum()))
            cost = (cc.w_b_q8 * led + cc.w_s_q8 * int(work_dec[k])) * sig + cc.w_q_us * int(m.sum()) * 65536
            if best is None or cost < best[0]:
                best = (cost, d)
        assert best[1] == idc[k], k


@pytest.mark.parametrize("cc", [
    W.CALIBRATED,
    W.CALIBRATED.replace(tau_dec_us=7600, tau_pre0_us=40000),      # a mispriced set
    W.CALIBRATED.replace(w_q_us=0, w_s_q8=0),                       # backlog only
], ids=["calibrated", "mispriced", "ledger_only"])
def test_proxy_backlog_rederived_from_outputs(orc, cc):
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2500, replica=2)
    cc = cc.replace(proxy_backlog=1, ablate=W.ABLATE_PRESSURE)
    res = orc.simulate(wl.sim, cc, W.POLICY_LEARNED, tr)
    assert res["status"] == 0
    _rederive(tr, res, wl.sim, cc)


def test_proxy_ledger_differs_from_true_backlog(orc):
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2500, replica=2)
    a = orc.simulate(wl.sim, W.CALIBRATED, W.POLICY_LEARNED, tr)
    b = orc.simulate(wl.sim, W.CALIBRATED.replace(proxy_backlog=1), W.POLICY_LEARNED, tr)
    assert a["status"] == b["status"] == 0
    assert not np.array_equal(a["i_dec"], b["i_dec"])


def test_proxy_ledger_with_unit_weights_is_the_length_heuristic(orc):
    """Ledger weight only, tau_pre = 0, tau_pre0 = tau_dec = 1: the prefill
    ledger is the in-flight count and the decode ledger the in-flight sum of
    predicted lengths -- the length heuristic with threshold 0."""
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2500, replica=4)
    cc = W.CostConsts(tau_pre0_us=1, tau_pre_us=0, tau_dec_us=1, w_q_us=0, w_b_q8=256, w_s_q8=0, rho_q8=0,
                      proxy_backlog=1)
    a = orc.simulate(wl.sim, cc, W.POLICY_LEARNED, tr)
    b = orc.simulate(wl.sim.replace(heuristic_threshold_tokens=0), W.CALIBRATED, W.POLICY_HEURISTIC, tr)
    assert a["status"] == b["status"] == 0
    for key in ("i_pre", "i_dec", "t_first_us", "t_done_us"):
        assert np.array_equal(a[key], b[key]), key


def test_proxy_ledger_is_invariant_to_the_unit_of_time(orc):
    """sec. III-B: with the backlog priced by the router's own constants, every
    term of the (pressure-free) cost is linear in (tau_pre0, tau_pre, tau_dec,
    w_q), so doubling all of them changes no decision; the true backlog is in
    real microseconds and does not scale with them."""
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2500, replica=7)
    base = W.CALIBRATED.replace(ablate=W.ABLATE_PRESSURE)
    dbl = base.replace(tau_pre0_us=2 * base.tau_pre0_us, tau_pre_us=2 * base.tau_pre_us,
                       tau_dec_us=2 * base.tau_dec_us, w_q_us=2 * base.w_q_us)
    pa = orc.simulate(wl.sim, base.replace(proxy_backlog=1), W.POLICY_LEARNED, tr)
    pb = orc.simulate(wl.sim, dbl.replace(proxy_backlog=1), W.POLICY_LEARNED, tr)
    assert pa["status"] == pb["status"] == 0 and pa["hash"] == pb["hash"]
    ta = orc.simulate(wl.sim, base, W.POLICY_LEARNED, tr)
    tb = orc.simulate(wl.sim, dbl, W.POLICY_LEARNED, tr)
    assert ta["status"] == tb["status"] == 0 and ta["hash"] != tb["hash"]


def _grid_trace(orc, wl, n, replica, grid):
    tr = orc.gen_trace(wl.trace, n, replica=replica)
    tr["arrival_us"] = (tr["arrival_us"] // grid) * grid
    return tr


@pytest.mark.parametrize("pol", [W.POLICY_LEARNED, W.POLICY_LEARNED_P2])
def test_poll_at_every_arrival_instant_is_live(orc, pol):
    """Arrivals on a 1 ms grid: a 1 ms poll samples the occupancy at every
    arrival instant, after that instant's events, which is the live value."""
    wl = W.replica_sweep()
    tr = _grid_trace(orc, wl, 2500, 3, 1000)
    a = orc.simulate(wl.sim, W.CALIBRATED, pol, tr)
    b = orc.simulate(wl.sim, W.CALIBRATED.replace(poll_us=1000), pol, tr)
    assert a["status"] == b["status"] == 0 and a["hash"] == b["hash"]


@pytest.mark.parametrize("pol", [W.POLICY_LEARNED, W.POLICY_LEARNED_P2])
def test_poll_never_refreshed_is_pressure_ablation(orc, pol):
    """A poll period beyond every arrival leaves only the poll at 0 (empty
    cluster): the post-admission pressure is the same on every decode
    candidate, so it cannot change an argmin -- the decisions of the pressure-
    ablated router."""
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2500, replica=3)
    a = orc.simulate(wl.sim, W.CALIBRATED.replace(poll_us=1 << 39), pol, tr)
    b = orc.simulate(wl.sim, W.CALIBRATED.replace(ablate=W.ABLATE_PRESSURE), pol, tr)
    assert a["status"] == b["status"] == 0 and a["hash"] == b["hash"]


def test_stale_occupancy_changes_routes_under_kv_scarcity(orc):
    """With a tight KV budget the pressure term matters, and a 50 ms-old view of
    it routes differently from the live one (sec. VI: the deployed signal)."""
    wl = W.large_pool(n_replicas=1, n_req=3000)
    tr = orc.gen_trace(wl.trace, 3000, replica=0)
    cc = wl.consts[0]
    a = orc.simulate(wl.sim, cc, W.POLICY_LEARNED, tr)
    b = orc.simulate(wl.sim, W.as_deployed(cc).replace(proxy_backlog=0), W.POLICY_LEARNED, tr)
    assert a["status"] == b["status"] == 0
    assert not np.array_equal(a["i_dec"], b["i_dec"])


def test_signal_bounds(orc):
    wl = W.single_replica()
    tr = orc.gen_trace(wl.trace, 50)
    for bad in (dict(proxy_backlog=2), dict(proxy_backlog=-1), dict(poll_us=-1), dict(poll_us=(1 << 39) + 1)):
        assert orc.simulate(wl.sim, W.CALIBRATED.replace(**bad), W.POLICY_LEARNED, tr)["status"] == -1
    assert orc.simulate(wl.sim, W.CALIBRATED.replace(poll_us=1 << 39, proxy_backlog=1), W.POLICY_LEARNED,
                        tr)["status"] == 0
