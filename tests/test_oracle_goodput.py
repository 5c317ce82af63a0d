"""Pins the oracle's goodput and nearest-rank P99: a hand-computed case and
numpy's inverted-CDF percentile (the nearest-rank definition); the same for P99 TPOT,
which a closed form of isolated requests also fixes."""
import numpy as np

from paper_2609_16206_gb300 import workloads as W


def test_hand_computed_goodput(orc):
    sc = W.SimCfg()          # class 0: TTFT 1 s, TPOT 100 ms; class 1: 5 s, 250 ms
    tr = {"arrival_us": np.array([0, 0, 0, 0, 0], np.int64), "true_out": np.array([1, 3, 3, 2, 11], np.int32),
          "slo_class": np.array([0, 0, 1, 0, 1], np.uint8)}
    t_first = np.array([1_000_000, 900_000, 4_000_000, 1_000_001, 100], np.int64)
    t_done = np.array([1_000_000, 1_100_000, 4_500_001, 1_100_000, 2_500_100], np.int64)
    # r0 TTFT = 1e6 met (o = 1); r1 TPOT 200000 <= 2 * 100000 met; r2 500001 > 2 * 250000 missed;
    # r3 TTFT 1000001 > 1e6 missed; r4 2500000 <= 10 * 250000 met -> 3
    met, p99 = orc.goodput(sc, tr, t_first, t_done)
    assert met == 3
    assert p99 == 4_000_000   # N = 5 -> sorted index ceil(4.95) - 1 = 4, the largest TTFT


def test_p99_is_nearest_rank(orc):
    rng = np.random.default_rng(3)
    sc = W.SimCfg()
    for n in (1, 2, 99, 100, 101, 2000, 20_000, 20_001):
        ttft = rng.integers(0, 10**9, n)
        tr = {"arrival_us": np.zeros(n, np.int64), "true_out": np.ones(n, np.int32),
              "slo_class": np.zeros(n, np.uint8)}
        _, p99 = orc.goodput(sc, tr, ttft, ttft)
        assert p99 == int(np.percentile(ttft, 99, method="inverted_cdf"))


def test_empty_row(orc):
    sc = W.SimCfg()
    z = np.zeros(0, np.int64)
    tr = {"arrival_us": z, "true_out": np.zeros(0, np.int32), "slo_class": np.zeros(0, np.uint8)}
    assert orc.goodput(sc, tr, z, z) == (0, -1)


def test_p99_tpot_hand_computed(orc):
    """TPOT = floor((t_done - t_first) / (o - 1)) over requests with o >= 2, nearest-rank P99."""
    tr = {"true_out": np.array([1, 3, 3, 2, 11], np.int32)}
    t_first = np.array([1_000_000, 900_000, 4_000_000, 1_000_001, 100], np.int64)
    t_done = np.array([1_000_000, 1_100_000, 4_500_001, 1_100_000, 2_500_100], np.int64)
    # r0 has one token (no TPOT); r1 200000 / 2 = 100000; r2 500001 / 2 = 250000.5 -> 250000;
    # r3 99999 / 1; r4 2500000 / 10 = 250000.  M = 4 -> sorted index ceil(3.96) - 1 = 3 -> 250000
    assert orc.p99_tpot(tr, t_first, t_done) == 250_000
    # the worked 1P+2D trace: r0 (o = 2) first token at 52,200 us, done at 67,400 us; r1 has one token
    assert orc.p99_tpot({"true_out": np.array([2, 1], np.int32)}, np.array([52_200, 87_200]),
                        np.array([67_400, 87_200])) == 15_200


def test_p99_tpot_is_nearest_rank(orc):
    rng = np.random.default_rng(11)
    for n in (1, 2, 100, 101, 2000, 20_001):
        o = rng.integers(1, 4097, n).astype(np.int32)
        o[rng.random(n) < 0.3] = 1
        tf = rng.integers(0, 10**9, n)
        td = tf + rng.integers(0, 10**8, n)
        sel = o >= 2
        want = -1 if not sel.any() else int(np.percentile((td - tf)[sel] // (o[sel].astype(np.int64) - 1), 99,
                                                          method="inverted_cdf"))
        assert orc.p99_tpot({"true_out": o}, tf, td) == want


def test_p99_tpot_no_multi_token_request(orc):
    z = np.zeros(0, np.int64)
    assert orc.p99_tpot({"true_out": np.zeros(0, np.int32)}, z, z) == -1
    ones = np.ones(5, np.int32)
    t = np.arange(5, dtype=np.int64)
    assert orc.p99_tpot({"true_out": ones}, t, t + 7) == -1


def test_p99_tpot_of_isolated_requests(orc):
    """Requests 10 s apart never share a batch: each decode step lasts 15,200 us plus the KV term
    floor((p + j) / 1000), so TPOT follows from the closed form, not from the simulator."""
    rng = np.random.default_rng(6)
    n = 40
    p = rng.integers(16, 8193, n).astype(np.int32)
    o = rng.integers(1, 401, n).astype(np.int32)
    tr = {"arrival_us": (np.arange(n, dtype=np.int64) * 10_000_000), "prompt_len": p, "true_out": o,
          "pred_out": o.copy(), "slo_class": np.zeros(n, np.uint8)}
    res = orc.simulate(W.SimCfg(n_prefill=1, n_decode=2), W.CALIBRATED, W.POLICY_RR, tr)
    assert res["status"] == 0
    tpots = sorted(sum(15_200 + (int(p[k]) + j) // 1000 for j in range(1, int(o[k]))) // (int(o[k]) - 1)
                   for k in range(n) if o[k] >= 2)
    want = tpots[-(-99 * len(tpots) // 100) - 1]
    assert orc.p99_tpot(tr, res["t_first_us"], res["t_done_us"]) == want
