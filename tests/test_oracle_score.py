"""Pins the oracle's fp64 brute-force scorer: hand-computed dyadic costs,
tie-breaking, invalid classes, and equivariance under instance permutation."""
import json
import os

import numpy as np

from conftest import GOLDEN
from paper_2609_16206_gb300 import workloads as W


def _hand():
    with open(os.path.join(GOLDEN, "score_hand.json")) as f:
        return json.load(f)


def test_hand_computed(orc):
    h = _hand()
    s, r, e = h["state"], h["requests"], h["expect"]
    am, best, second = orc.score_batch(r["p"], r["oh"], np.array(r["cls"], np.uint8), s["Q"], s["A"], s["kappa"],
                                       h["consts"])
    assert am.tolist() == e["argmin"]
    for i, b in enumerate(e["best"]):
        if b is None:
            assert np.isnan(best[i]) and np.isnan(second[i])
        else:
            assert best[i] == b and second[i] == e["second"][i]
    for i, row in enumerate(e["all_costs"]):
        got = orc.score_pairs(r["p"], r["oh"], np.array(r["cls"], np.uint8), [i] * 4, [0, 1, 2, 3],
                              s["Q"], s["A"], s["kappa"], h["consts"])
        assert got.tolist() == row


def test_single_instance(orc):
    p, oh, cls = W.score_requests(1000)
    Q, A, kap = W.score_state(1)
    am, best, second = orc.score_batch(p, oh, cls, Q, A, kap, W.SCORE_CONSTS)
    assert np.all(am == 0) and np.all(np.isinf(second))


def test_permutation_equivariance(orc):
    p, oh, cls = W.score_requests(4000, seed=9)
    Q, A, kap = W.score_state(64, seed=10)
    am, best, _ = orc.score_batch(p, oh, cls, Q, A, kap, W.SCORE_CONSTS)
    perm = np.random.default_rng(2).permutation(64)
    am2, best2, _ = orc.score_batch(p, oh, cls, Q[perm], A[perm], kap[perm], W.SCORE_CONSTS)
    assert np.array_equal(perm[am2], am)
    assert np.array_equal(best, best2)


def test_monotone_in_queue(orc):
    p, oh, cls = W.score_requests(500, seed=4)
    Q, A, kap = W.score_state(8, seed=5)
    _, best, _ = orc.score_batch(p, oh, cls, Q, A, kap, W.SCORE_CONSTS)
    _, best2, _ = orc.score_batch(p, oh, cls, Q + 1000, A, kap, W.SCORE_CONSTS)
    assert np.all(best2 > best)
