"""Checkpoint / resume of sweeps by replica range (host logic, no GPU): a fake
chunk runner stands in for the GPU, failures are injected on the host (a run
that raises mid-sweep, a stop after a few chunks, an append cut short), and
the resumed sweep must equal one uninterrupted run, simulating every chunk
exactly once."""
import json

import numpy as np
import pytest

from paper_2609_16206_gb300 import sweep
from paper_2609_16206_gb300 import workloads as W

WL = W.replica_sweep(n_replicas=10, n_req=100)
ROWS_PER_REPLICA = len(WL.consts) * len(WL.policies)


def fake_rows(off, cnt):
    """Deterministic per-row results of replicas [off, off + cnt), as a function of the row index alone."""
    rows = range(off * ROWS_PER_REPLICA, (off + cnt) * ROWS_PER_REPLICA)
    return {"row_hash": [(0x9E3779B97F4A7C15 * (r + 1)) & ((1 << 64) - 1) for r in rows],
            "row_status": [0 if r % 7 else -3 for r in rows],
            "met": [r * 3 for r in rows], "p99_ttft_us": [1000 + r for r in rows]}


class Runner:
    def __init__(self, fail_at=None):
        self.calls = []
        self.fail_at = fail_at

    def __call__(self, off, cnt):
        if self.fail_at is not None and len(self.calls) == self.fail_at:
            raise RuntimeError("rank lost")  # injected on the host
        self.calls.append((off, cnt))
        return fake_rows(off, cnt)


def reference():
    return fake_rows(0, WL.n_replicas)


def same(res):
    ref = reference()
    return all(np.array_equal(res[k], np.asarray(ref[k], dtype=res[k].dtype)) for k in sweep.RESULT_FIELDS)


def test_uninterrupted_run(tmp_path):
    run = Runner()
    res = sweep.resumable_sweep(WL, str(tmp_path / "j"), chunk=3, run_chunk=run)
    assert same(res)
    assert run.calls == [(0, 3), (3, 3), (6, 3), (9, 1)]


def test_stop_and_resume(tmp_path):
    j = str(tmp_path / "j")
    first = Runner()
    assert sweep.resumable_sweep(WL, j, chunk=3, run_chunk=first, max_chunks=2) is None
    assert first.calls == [(0, 3), (3, 3)]
    second = Runner()
    res = sweep.resumable_sweep(WL, j, chunk=3, run_chunk=second)
    assert second.calls == [(6, 3), (9, 1)]  # journaled chunks are not simulated again
    assert same(res)
    third = Runner()
    assert same(sweep.resumable_sweep(WL, j, chunk=3, run_chunk=third)) and third.calls == []


def test_failure_mid_sweep_then_resume(tmp_path):
    j = str(tmp_path / "j")
    with pytest.raises(RuntimeError):
        sweep.resumable_sweep(WL, j, chunk=4, run_chunk=Runner(fail_at=1))
    assert len(open(j).read().splitlines()) == 1  # the chunk finished before the failure is kept
    again = Runner()
    assert same(sweep.resumable_sweep(WL, j, chunk=4, run_chunk=again))
    assert again.calls == [(4, 4), (8, 2)]


def test_append_cut_short_is_ignored_and_repaired(tmp_path):
    j = tmp_path / "j"
    sweep.resumable_sweep(WL, str(j), chunk=5, run_chunk=Runner(), max_chunks=1)
    with open(j, "a") as f:  # a write killed half way: no newline
        f.write('{"fingerprint": "x", "offset": 5, "row_ha')
    again = Runner()
    assert same(sweep.resumable_sweep(WL, str(j), chunk=5, run_chunk=again))
    assert again.calls == [(5, 5)]
    lines = open(j).read().splitlines()
    assert len(lines) == 2 and all(json.loads(line)["count"] == 5 for line in lines)


def test_journal_of_another_sweep_is_refused(tmp_path):
    j = str(tmp_path / "j")
    sweep.resumable_sweep(WL, j, chunk=5, run_chunk=Runner(), max_chunks=1)
    with pytest.raises(ValueError):
        sweep.resumable_sweep(WL, j, chunk=4, run_chunk=Runner())  # other chunking
    other = W.replica_sweep(n_replicas=10, n_req=101)
    with pytest.raises(ValueError):
        sweep.resumable_sweep(other, j, chunk=5, run_chunk=Runner())


def test_corrupt_line_inside_the_journal_raises(tmp_path):
    j = tmp_path / "j"
    sweep.resumable_sweep(WL, str(j), chunk=5, run_chunk=Runner(), max_chunks=1)
    text = open(j).read()
    open(j, "w").write("{not json}\n" + text)
    with pytest.raises(ValueError):
        sweep.resumable_sweep(WL, str(j), chunk=5, run_chunk=Runner())


def test_no_replicas(tmp_path):
    empty = W.replica_sweep(n_replicas=0, n_req=100)
    run = Runner()
    res = sweep.resumable_sweep(empty, str(tmp_path / "j"), chunk=3, run_chunk=run)
    assert run.calls == [] and all(res[k].size == 0 for k in sweep.RESULT_FIELDS)
