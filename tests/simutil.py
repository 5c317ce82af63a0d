"""Helpers shared by the simulator tests: fixtures from tests/golden and
re-derivations of queue signals from a row's outputs."""
import json
import os

import numpy as np

from conftest import GOLDEN
from paper_2609_16206_gb300 import workloads as W


def worked_traces():
    with open(os.path.join(GOLDEN, "worked_traces.json")) as f:
        return json.load(f)["traces"]


def sim_from(d, **kw):
    base = dict(n_classes=2, ttft_slo_us=(1_000_000, 5_000_000), tpot_slo_us=(100_000, 250_000))
    base.update(d)
    base.update(kw)
    return W.SimCfg(**base)


def consts_from(d):
    if d is None:
        return W.CALIBRATED
    d = dict(d)
    d["sigma_q8"] = tuple(d["sigma_q8"])
    return W.CostConsts(**d)


def trace_from(d):
    return {"arrival_us": np.array(d["arrival_us"], np.int64), "prompt_len": np.array(d["prompt_len"], np.int32),
            "true_out": np.array(d["true_out"], np.int32), "pred_out": np.array(d["pred_out"], np.int32),
            "slo_class": np.array(d["slo_class"], np.uint8)}


def inflight_counts(t, owner, finish, n_inst, k):
    """#{j < k : owner[j] == i and finish[j] > t} per instance i."""
    m = (owner[:k] >= 0) & (finish[:k] > t)
    return np.bincount(owner[:k][m], minlength=n_inst)


def inflight_sums(t, owner, finish, weight, n_inst, k):
    m = finish[:k] > t
    return np.bincount(owner[:k][m], weights=weight[:k][m].astype(np.float64), minlength=n_inst)
