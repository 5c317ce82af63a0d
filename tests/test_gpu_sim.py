"""Parity: the GPU replica simulator matches the CPU oracle bit for bit --
every routing decision, first-token and completion time, and the row hash --
on hand-made traces, generated workloads, several constant sets, the widest
pool, ragged and empty inputs, and the error paths."""
import numpy as np
import pytest
import torch

import simutil as U
from gpuutil import gen, host_trace, need_gpu, simulate, to_dev
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _check_rows(orc, sc, sets, pols, tr_host_rows, res, n_req, full=True):
    row = 0
    for r, trh in enumerate(tr_host_rows):
        for cc in sets:
            for pol in pols:
                o = orc.simulate(sc, cc, pol, trh)
                assert res["status"][row] == o["status"], (row, res["status"][row], o["status"])
                if o["status"] == 0:
                    assert int(res["hash"][row]) == o["hash"], row
                    if full:
                        for key in ("t_first_us", "t_done_us", "i_pre", "i_dec"):
                            if key in res:
                                got, want = res[key][row], o[key]
                                assert np.array_equal(got, want), (key, row, np.flatnonzero(got != want)[:5])
                row += 1


@pytest.mark.parametrize("case", U.worked_traces(), ids=lambda c: c["name"])
def test_worked_traces(orc, case):
    ctr = need_gpu()
    sc = U.sim_from(case["sim"])
    trh = U.trace_from(case["requests"])
    sets = [U.consts_from(case["consts"])]
    res = simulate(ctr, sc, sets, list(W.ALL_POLICIES), to_dev(trh), 1, trh["arrival_us"].size)
    _check_rows(orc, sc, sets, list(W.ALL_POLICIES), [trh], res, trh["arrival_us"].size)
    # and the hand-derived values themselves
    j = list(W.ALL_POLICIES).index(case["policy"])
    for key in ("t_first_us", "t_done_us", "i_pre", "i_dec"):
        if key in case["expect"]:
            assert res[key][j].tolist() == case["expect"][key]


def test_single_replica_all_policies(orc):
    ctr = need_gpu()
    wl = W.single_replica()
    tr = gen(ctr, wl.trace, 1, wl.n_req)
    res = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, 1, wl.n_req)
    _check_rows(orc, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), [host_trace(tr, 0)], res, wl.n_req)


def test_bursty_replicas_all_policies(orc):
    ctr = need_gpu()
    wl = W.replica_sweep()
    R, N = 20, 3000
    tr = gen(ctr, wl.trace, R, N)
    res = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, R, N)
    _check_rows(orc, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), [host_trace(tr, r) for r in range(R)], res, N)


def test_mispriced_constant_sets(orc):
    ctr = need_gpu()
    wl = W.replica_sweep()
    sets = W.mispriced_sets()[::9]
    R, N = 3, 1500
    tr = gen(ctr, wl.trace, R, N)
    res = simulate(ctr, wl.sim, sets, [W.POLICY_LEARNED, W.POLICY_JSQ], tr, R, N)
    _check_rows(orc, wl.sim, sets, [W.POLICY_LEARNED, W.POLICY_JSQ], [host_trace(tr, r) for r in range(R)], res, N)


def test_large_pool_overload(orc):
    """4P+28D (all 32 lanes) at prefill overload: deep queues, three classes."""
    ctr = need_gpu()
    wl = W.large_pool(rate_mreq=34_000)
    R, N = 2, 4000
    tr = gen(ctr, wl.trace, R, N)
    cc = wl.consts[0]
    res = simulate(ctr, wl.sim, [cc], list(W.ALL_POLICIES), tr, R, N)
    _check_rows(orc, wl.sim, [cc], list(W.ALL_POLICIES), [host_trace(tr, r) for r in range(R)], res, N)


@pytest.mark.parametrize("n_pre,n_dec", [(1, 1), (31, 1), (1, 31), (3, 5)])
def test_pool_shapes(orc, n_pre, n_dec):
    ctr = need_gpu()
    sc = W.SimCfg(n_prefill=n_pre, n_decode=n_dec)
    tc = W.TraceCfg(rate_mreq=(3000, 3000), seed=n_pre * 100 + n_dec)
    N = 700
    tr = gen(ctr, tc, 2, N)
    res = simulate(ctr, sc, [W.CALIBRATED], list(W.ALL_POLICIES), tr, 2, N)
    _check_rows(orc, sc, [W.CALIBRATED], list(W.ALL_POLICIES), [host_trace(tr, r) for r in range(2)], res, N)


@pytest.mark.parametrize("N", [0, 1, 31, 33, 65])
def test_ragged_and_empty(orc, N):
    ctr = need_gpu()
    wl = W.replica_sweep()
    tr = gen(ctr, wl.trace, 2, N)
    res = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, 2, N)
    _check_rows(orc, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), [host_trace(tr, r) for r in range(2)], res, N)


def test_small_workspace_same_results(orc):
    """A workspace with room for only two warp slots runs the rows in turn."""
    ctr = need_gpu()
    wl = W.replica_sweep()
    R, N = 6, 800
    tr = gen(ctr, wl.trace, R, N)
    full = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, R, N)
    slot = ctr.ctr_workspace_bytes(0, wl.sim, 1, N) - 256
    small = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, R, N, ws_bytes=256 + 2 * slot)
    for key in full:
        assert np.array_equal(full[key], small[key]), key


def test_routes_optional(orc):
    ctr = need_gpu()
    wl = W.replica_sweep()
    tr = gen(ctr, wl.trace, 2, 500)
    a = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, 2, 500, routes=False)
    b = simulate(ctr, wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, 2, 500)
    assert np.array_equal(a["hash"], b["hash"]) and np.array_equal(a["t_done_us"], b["t_done_us"])


def test_capacity_overflow_matches_oracle(orc):
    ctr = need_gpu()
    wl = W.replica_sweep()
    N = 2000
    tr = gen(ctr, wl.trace, 1, N)
    trh = host_trace(tr, 0)
    st = orc.simulate(wl.sim, W.CALIBRATED, W.POLICY_LEARNED, trh)["stats"]
    caps = dict(cap_pending=st["max_pending"], cap_waiting=st["max_waiting"], cap_active=st["max_active"],
                cap_prefill_ring=st["max_prefill"])
    ok = simulate(ctr, wl.sim.replace(**caps), [W.CALIBRATED], [W.POLICY_LEARNED], tr, 1, N)
    assert ok["status"][0] == 0
    for name in caps:
        if caps[name] <= 1:
            continue
        tight = dict(caps)
        tight[name] -= 1
        bad = simulate(ctr, wl.sim.replace(**tight), [W.CALIBRATED], [W.POLICY_LEARNED], tr, 1, N)
        assert bad["status"][0] == ctr.CTR_EOVERFLOW, name


def test_step_budget_and_invalid_rows(orc):
    ctr = need_gpu()
    wl = W.single_replica()
    N = 300
    trh = orc.gen_trace(wl.trace, N)
    res = simulate(ctr, wl.sim.replace(max_steps_per_instance=50), [W.CALIBRATED], [W.POLICY_RR], to_dev(trh), 1, N)
    assert res["status"][0] == ctr.CTR_ETIMEOUT
    bad = dict(trh)
    bad["true_out"] = trh["true_out"].copy()
    bad["true_out"][7] = 0
    rows = {k: np.stack([trh[k], bad[k]]) for k in trh}
    res = simulate(ctr, wl.sim, [W.CALIBRATED], [W.POLICY_LEARNED], to_dev(rows), 2, N)
    assert res["status"].tolist() == [0, ctr.CTR_EINVAL]
    assert int(res["hash"][0]) == orc.simulate(wl.sim, W.CALIBRATED, 0, trh)["hash"]
    un = dict(trh)
    un["arrival_us"] = trh["arrival_us"].copy()
    un["arrival_us"][40] = un["arrival_us"][39] - 1
    assert simulate(ctr, wl.sim, [W.CALIBRATED], [0], to_dev(un), 1, N)["status"][0] == ctr.CTR_EINVAL


def test_host_validation_rejects(orc):
    ctr = need_gpu()
    wl = W.single_replica()
    tr = gen(ctr, wl.trace, 1, 50)
    for sc, sets, pols in ((wl.sim.replace(n_prefill=0), [W.CALIBRATED], [0]),
                           (wl.sim.replace(n_prefill=20, n_decode=13), [W.CALIBRATED], [0]),
                           (wl.sim, [W.CALIBRATED.replace(w_b_q8=1024)], [0]),
                           (wl.sim, [W.CALIBRATED], [5]),
                           (wl.sim, [W.CALIBRATED.replace(ablate=8)], [0]),
                           (wl.sim, [W.CALIBRATED], []),
                           (wl.sim.replace(cap_active=0), [W.CALIBRATED], [0])):
        with pytest.raises(Exception):
            simulate(ctr, sc, sets, pols, tr, 1, 50)


def test_full_size_sweep_sampled(orc):
    """The benchmarked configuration in the benchmark's launch shape: 4,096 bursty
    replicas x 20,000 requests x 4 policies in one launch; sampled rows against
    the oracle by hash (every row's status must be OK)."""
    ctr = need_gpu()
    wl = W.replica_sweep()
    R, N = wl.n_replicas, wl.n_req
    tr = gen(ctr, wl.trace, R, N)
    rows = R * 4
    tf = torch.empty((rows, N), dtype=torch.int64, device="cuda")
    td = torch.empty_like(tf)
    h = torch.empty(rows, dtype=torch.int64, device="cuda")
    st = torch.empty(rows, dtype=torch.int32, device="cuda")
    ws = ctr.simulate_workspace(wl.sim, rows, N, "cuda")
    ctr.ctr_simulate(wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, R, N, tf, td, h, st, ws)
    torch.cuda.synchronize()
    assert int((st != 0).sum()) == 0
    hh = h.cpu().numpy().astype(np.uint64)
    for r in (0, 1, 2, 5, 97, 511, 1024, 1366, 2048, 2731, 3000, 3333, 3500, 4000, 4094, 4095):  # all 3 seeds
        trh = host_trace(tr, r)
        for j, pol in enumerate(W.ALL_POLICIES):
            o = orc.simulate(wl.sim, W.CALIBRATED, pol, trh)
            assert o["status"] == 0 and int(hh[r * 4 + j]) == o["hash"], (r, pol)


@pytest.mark.parametrize("ablate", [1, 2, 4, 7])
def test_feature_ablation(orc, ablate):
    ctr = need_gpu()
    wl = W.replica_sweep()
    R, N = 6, 2000
    tr = gen(ctr, wl.trace, R, N)
    cc = W.CALIBRATED.replace(ablate=ablate)
    res = simulate(ctr, wl.sim, [cc], [W.POLICY_LEARNED, W.POLICY_LEARNED_P2], tr, R, N)
    _check_rows(orc, wl.sim, [cc], [W.POLICY_LEARNED, W.POLICY_LEARNED_P2], [host_trace(tr, r) for r in range(R)],
                res, N)


@pytest.mark.parametrize("wl", [W.replica_sweep(), W.large_pool(rate_mreq=34_000), W.single_replica()],
                         ids=["2p6d", "4p28d", "1p3d"])
def test_power_of_two_router(orc, wl):
    ctr = need_gpu()
    R, N = 4, 2500
    tr = gen(ctr, wl.trace, R, N)
    pols = [W.POLICY_LEARNED_P2, W.POLICY_LEARNED, W.POLICY_RR]
    res = simulate(ctr, wl.sim, [wl.consts[0]], pols, tr, R, N)
    _check_rows(orc, wl.sim, [wl.consts[0]], pols, [host_trace(tr, r) for r in range(R)], res, N)


def _signal_sets(base):
    """True / ledger backlog x live / 50 ms / 7 ms occupancy, plus a mispriced ledger set."""
    return [base, base.replace(proxy_backlog=1), base.replace(poll_us=W.PROXY_POLL_US), W.as_deployed(base),
            base.replace(poll_us=7_000, proxy_backlog=1, ablate=W.ABLATE_PREDICTED_LENGTH),
            W.as_deployed(base).replace(tau_dec_us=base.tau_dec_us // 2, tau_pre0_us=2 * base.tau_pre0_us)]


@pytest.mark.parametrize("wl", [W.replica_sweep(), W.large_pool(rate_mreq=34_000), W.single_replica()],
                         ids=["2p6d", "4p28d", "1p3d"])
def test_proxy_signals(orc, wl):
    """Ledger backlog and polled occupancy (sec. IV-A) in one launch with the
    true signals, every row bit-identical to the oracle."""
    ctr = need_gpu()
    R, N = 3, 2500
    tr = gen(ctr, wl.trace, R, N)
    sets = _signal_sets(wl.consts[0])
    pols = [W.POLICY_LEARNED, W.POLICY_LEARNED_P2]
    res = simulate(ctr, wl.sim, sets, pols, tr, R, N)
    _check_rows(orc, wl.sim, sets, pols, [host_trace(tr, r) for r in range(R)], res, N)


def test_proxy_signals_host_validation():
    ctr = need_gpu()
    wl = W.single_replica()
    tr = gen(ctr, wl.trace, 1, 16)
    for bad in (dict(proxy_backlog=2), dict(poll_us=-1), dict(poll_us=(1 << 39) + 1)):
        with pytest.raises(ctr.CtrError):
            simulate(ctr, wl.sim, [W.CALIBRATED.replace(**bad)], [W.POLICY_LEARNED], tr, 1, 16)


ALL_FIVE = [W.POLICY_LEARNED, W.POLICY_RR, W.POLICY_JSQ, W.POLICY_HEURISTIC, W.POLICY_LEARNED_P2]


@pytest.mark.parametrize("budget", [900, 8192, 1 << 20])
def test_batched_prefill_document(orc, budget):
    """Batched prefill (sec. VI) on the Table 1 document workload, every policy."""
    ctr = need_gpu()
    wl = W.document(rate_mreq=6_500, batch_tokens=budget)
    R, N = 3, 2000
    tr = gen(ctr, wl.trace, R, N)
    res = simulate(ctr, wl.sim, [W.CALIBRATED], ALL_FIVE, tr, R, N)
    _check_rows(orc, wl.sim, [W.CALIBRATED], ALL_FIVE, [host_trace(tr, r) for r in range(R)], res, N)


def test_batched_prefill_equal_times(orc):
    """Arrivals on a 10 ms grid and batches of constant length 20 ms: arrivals
    land on batch ends all the time (the batch that starts there must not take
    them), with the proxy signals on as well."""
    ctr = need_gpu()
    wl = W.replica_sweep()
    R, N = 3, 2000
    tr = gen(ctr, wl.trace.replace(rate_mreq=(20_000, 60_000)), R, N)
    tr["arrival_us"].copy_((tr["arrival_us"] // 10_000) * 10_000)
    torch.cuda.synchronize()
    sc = wl.sim.replace(pre_us_per_tok=0, prefill_batch_tokens=3000, n_prefill=3, n_decode=5)
    sets = [W.CALIBRATED, W.as_deployed(W.CALIBRATED)]
    res = simulate(ctr, sc, sets, ALL_FIVE, tr, R, N)
    _check_rows(orc, sc, sets, ALL_FIVE, [host_trace(tr, r) for r in range(R)], res, N)


@pytest.mark.parametrize("caps", [dict(cap_prefill_ring=24), dict(cap_pending=12), dict(cap_waiting=2),
                                  dict(cap_active=20)], ids=lambda c: list(c)[0])
def test_batched_prefill_capacity_errors(orc, caps):
    ctr = need_gpu()
    wl = W.document(rate_mreq=9_000)
    R, N = 3, 1500
    tr = gen(ctr, wl.trace, R, N)
    sc = wl.sim.replace(**caps)
    res = simulate(ctr, sc, [W.CALIBRATED], ALL_FIVE, tr, R, N)
    _check_rows(orc, sc, [W.CALIBRATED], ALL_FIVE, [host_trace(tr, r) for r in range(R)], res, N)
    assert (res["status"] == -3).any()


@pytest.mark.parametrize("wl", [W.chat(), W.reasoning(), W.large_pool(rate_mreq=34_000)], ids=["chat", "reasoning", "4p28d"])
def test_workload_families_batched_prefill(orc, wl):
    ctr = need_gpu()
    R, N = 2, 2000
    tr = gen(ctr, wl.trace, R, N)
    sc = wl.sim.replace(prefill_batch_tokens=W.PREFILL_BATCH_TOKENS)
    sets = [wl.consts[0], W.as_deployed(wl.consts[0])]
    res = simulate(ctr, sc, sets, ALL_FIVE, tr, R, N)
    _check_rows(orc, sc, sets, ALL_FIVE, [host_trace(tr, r) for r in range(R)], res, N)


def _full_size_sampled(orc, wl, sets, samples):
    ctr = need_gpu()
    R, N = wl.n_replicas, wl.n_req
    pols = list(W.ALL_POLICIES)
    tr = gen(ctr, wl.trace, R, N)
    rows = R * len(sets) * len(pols)
    tf = torch.empty((rows, N), dtype=torch.int64, device="cuda")
    td = torch.empty_like(tf)
    h = torch.empty(rows, dtype=torch.int64, device="cuda")
    st = torch.empty(rows, dtype=torch.int32, device="cuda")
    ws = ctr.simulate_workspace(wl.sim, rows, N, "cuda")
    ctr.ctr_simulate(wl.sim, sets, pols, tr, R, N, tf, td, h, st, ws)
    torch.cuda.synchronize()
    assert int((st != 0).sum()) == 0
    hh = h.cpu().numpy().astype(np.uint64)
    for r in samples:
        trh = host_trace(tr, r)
        for si, cc in enumerate(sets):
            for j, pol in enumerate(pols):
                o = orc.simulate(wl.sim, cc, pol, trh)
                assert o["status"] == 0 and int(hh[(r * len(sets) + si) * len(pols) + j]) == o["hash"], (r, si, pol)


def test_full_size_document_batched_prefill_sampled(orc):
    """4,096 document replicas x 10,000 requests with batched prefill, one launch of the
    extended kernel; sampled rows against the oracle."""
    _full_size_sampled(orc, W.document(n_replicas=4096), [W.CALIBRATED], (0, 1, 2047, 4095))


def test_full_size_deployed_signals_sampled(orc):
    """The benchmarked sweep under the deployed proxy's signals (ledger backlog, 50 ms
    occupancy poll) beside the true ones, 4,096 x 20,000 in one launch; sampled rows."""
    _full_size_sampled(orc, W.replica_sweep(), [W.CALIBRATED, W.as_deployed(W.CALIBRATED)], (0, 3, 4095))
