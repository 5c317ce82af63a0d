"""Pins the oracle's goodput and nearest-rank P99: a hand-computed case and
numpy's inverted-CDF percentile (the nearest-rank definition)."""
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
