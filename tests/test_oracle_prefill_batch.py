"""Pins for batched prefill (sec. VI: continuous batching in both stages) and
the Table 1 workload families.  The prefill stage depends only on arrivals,
prompt lengths and the routing, so it is replayed here from scratch, in
Python, and compared with the oracle's prefill end and KV-ready times; the
learned router's batched backlog is re-derived from the same replay."""
from collections import deque

import numpy as np
import pytest

from paper_2609_16206_gb300 import workloads as W

B_CLAMP = 1 << 40


class _Prefill:
    """One prefill instance: the running batch's end (None = idle) and the queue."""

    def __init__(self):
        self.run_end = None
        self.queue = deque()


class _Replay:
    def __init__(self, sc, p):
        self.sc, self.p = sc, p
        self.inst = [_Prefill() for _ in range(sc.n_prefill)]
        self.pre_end = np.full(p.size, -1, np.int64)

    def _start(self, x, s):
        budget = self.sc.prefill_batch_tokens
        members = [x.queue.popleft()]
        tokens = int(self.p[members[0]])
        while x.queue and tokens + int(self.p[x.queue[0]]) <= budget:
            j = x.queue.popleft()
            members.append(j)
            tokens += int(self.p[j])
        x.run_end = s + self.sc.pre_base_us + self.sc.pre_us_per_tok * tokens
        for j in members:
            self.pre_end[j] = x.run_end

    def advance(self, t):
        """Every batch end at or before t; the next batch starts at that end
        with the queue as it was then (arrivals at t come after)."""
        for x in self.inst:
            while x.run_end is not None and x.run_end <= t:
                e = x.run_end
                x.run_end = None
                if x.queue:
                    self._start(x, e)

    def drain(self, i, t):
        """Time to serve everything queued or running on instance i."""
        x = self.inst[i]
        b = x.run_end - t if x.run_end is not None and x.run_end > t else 0
        q = list(x.queue)
        m = 0
        while m < len(q):
            tokens = int(self.p[q[m]])
            m += 1
            while m < len(q) and tokens + int(self.p[q[m]]) <= self.sc.prefill_batch_tokens:
                tokens += int(self.p[q[m]])
                m += 1
            b += self.sc.pre_base_us + self.sc.pre_us_per_tok * tokens
        return min(b, B_CLAMP)

    def route(self, k, t, i):
        x = self.inst[i]
        x.queue.append(k)
        if x.run_end is None:
            self._start(x, t)


def _replay_row(sc, tr, res, check_backlog_argmin=False):
    t = tr["arrival_us"].astype(np.int64)
    p = tr["prompt_len"].astype(np.int64)
    rp = _Replay(sc, p)
    for k in range(t.size):
        tk = int(t[k])
        rp.advance(tk)
        if check_backlog_argmin:
            b = [rp.drain(i, tk) for i in range(sc.n_prefill)]
            assert int(np.argmin(b)) == int(res["i_pre"][k]), k
        rp.route(k, tk, int(res["i_pre"][k]))
    rp.advance(1 << 62)
    assert np.array_equal(rp.pre_end, res["pre_end_us"])
    assert np.array_equal(rp.pre_end + sc.xfer_us_per_tok * p, res["t_ready_us"])


@pytest.mark.parametrize("wl", [W.replica_sweep(), W.single_replica(), W.document()], ids=lambda w: w.name[:8])
def test_budget_of_one_token_is_serial_prefill(orc, wl):
    """Prompts are >= 16 tokens, so a 1-token budget admits only the head:
    every batch is one request and the event-driven batches must reproduce the
    serial closed form (start = max(arrival, busy)) exactly, for every policy."""
    tr = orc.gen_trace(wl.trace, 2500, replica=1)
    sc = wl.sim.replace(prefill_batch_tokens=0)
    for pol in (W.POLICY_LEARNED, W.POLICY_RR, W.POLICY_JSQ, W.POLICY_HEURISTIC, W.POLICY_LEARNED_P2):
        a = orc.simulate(sc, W.CALIBRATED, pol, tr)
        b = orc.simulate(sc.replace(prefill_batch_tokens=1), W.CALIBRATED, pol, tr)
        assert a["status"] == b["status"] == 0
        assert a["hash"] == b["hash"], pol
        assert np.array_equal(a["pre_end_us"], b["pre_end_us"])


@pytest.mark.parametrize("budget", [900, 4096, 8192, 1 << 20])
@pytest.mark.parametrize("pol", [W.POLICY_RR, W.POLICY_JSQ, W.POLICY_LEARNED])
def test_prefill_schedule_replayed(orc, budget, pol):
    wl = W.document(rate_mreq=6_500)
    tr = orc.gen_trace(wl.trace, 2000, replica=3)
    sc = wl.sim.replace(prefill_batch_tokens=budget)
    res = orc.simulate(sc, W.CALIBRATED, pol, tr)
    assert res["status"] == 0
    _replay_row(sc, tr, res)
    sizes = np.unique(np.stack([res["i_pre"], res["pre_end_us"]]), axis=1, return_counts=True)[1]
    if budget >= 8192:
        assert sizes.max() > 1           # the overloaded document workload does form batches


def test_batched_backlog_rederived(orc):
    """Learned router with only the backlog weight: every prefill choice is the
    argmin of the replayed drain time (rest of the running batch plus the
    queue cut into budget-limited batches)."""
    wl = W.document(rate_mreq=6_500)
    tr = orc.gen_trace(wl.trace, 2000, replica=4)
    sc = wl.sim.replace(n_prefill=3, prefill_batch_tokens=4096)
    cc = W.CostConsts(w_q_us=0, w_s_q8=0, w_b_q8=256, sigma_q8=(256, 256, 256, 256))
    res = orc.simulate(sc, cc, W.POLICY_LEARNED, tr)
    assert res["status"] == 0
    _replay_row(sc, tr, res, check_backlog_argmin=True)
    assert np.bincount(res["i_pre"], minlength=3).min() > 100


def test_batched_prefill_queue_counts_running_members(orc):
    """JSQ counts a request on its prefill instance until its batch ends."""
    wl = W.document(rate_mreq=6_500)
    tr = orc.gen_trace(wl.trace, 1500, replica=5)
    sc = wl.sim.replace(n_prefill=3, prefill_batch_tokens=8192)
    res = orc.simulate(sc, W.CALIBRATED, W.POLICY_JSQ, tr)
    assert res["status"] == 0
    t, ip, end = tr["arrival_us"], res["i_pre"], res["pre_end_us"]
    for k in range(t.size):
        q = np.bincount(ip[:k][end[:k] > t[k]], minlength=3)
        assert int(np.argmin(q)) == int(ip[k]), k


def test_document_family_laws(orc):
    wl = W.document()
    tr = orc.gen_trace(wl.trace, 20_000, replica=0)
    p, o = tr["prompt_len"], tr["true_out"]
    assert p.min() >= 16 and p.max() == 4096
    assert 1900 < p.mean() < 2500                      # lognormal(ln 2048, 0.5), clipped at 4096
    assert np.median(o) < 200 and o.max() <= 4096       # short component only
    ch = orc.gen_trace(W.chat().trace, 20_000, replica=0)
    rs = orc.gen_trace(W.reasoning().trace, 20_000, replica=0)
    assert np.median(ch["true_out"]) < 200 < 700 < np.median(rs["true_out"])
    assert np.array_equal(ch["prompt_len"], rs["prompt_len"])   # same prompt law and stream


def test_batch_budget_bounds(orc):
    wl = W.single_replica()
    tr = orc.gen_trace(wl.trace, 50)
    for bad in (-1, (1 << 30) + 1):
        assert orc.simulate(wl.sim.replace(prefill_batch_tokens=bad), W.CALIBRATED, 0, tr)["status"] == -1
