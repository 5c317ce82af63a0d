"""Multi-GPU partitioning of the replica sweep, exercised on the CPU: the
replica sets of the ranks are disjoint and cover the sweep, and results do
not depend on the partition.  World size 2 with the gloo backend; each rank
runs the oracle on its own replicas (no data-path collective), then the
results are gathered only to compare them with a single-process run."""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_16206_gb300 import sweep
from paper_2609_16206_gb300 import workloads as W

N_REQ = 400
PER_RANK = 2


def test_shard_split_covers_disjointly():
    for total in (0, 1, 5, 4096, 4097):
        for world in (1, 2, 3, 8):
            seen = []
            for r in range(world):
                off, cnt = sweep.shard_split(total, world, r)
                seen.extend(range(off, off + cnt))
            assert seen == list(range(total))


def test_weak_shards_are_disjoint():
    blocks = [set(range(*(lambda o, c: (o, o + c))(*sweep.shard(r, 4096)))) for r in range(8)]
    for i in range(8):
        for j in range(i + 1, 8):
            assert not blocks[i] & blocks[j]


def _rows(replicas):
    import oracle
    wl = W.replica_sweep()
    out = {}
    for g in replicas:
        tr = oracle.gen_trace(wl.trace, N_REQ, replica=g)
        for pol in W.ALL_POLICIES:
            res = oracle.simulate(wl.sim, W.CALIBRATED, pol, tr)
            out[(g, pol)] = (res["status"], res["hash"])
    return out


def _worker(rank, world, port, queue):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        off, cnt = sweep.shard(rank, PER_RANK)
        mine = _rows(range(off, off + cnt))
        gathered = [None] * world
        dist.all_gather_object(gathered, mine)
        if rank == 0:
            queue.put(gathered)
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_rank_sweep_matches_single_process():
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    world = 2
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, queue)) for r in range(world)]
    for p in procs:
        p.start()
    gathered = queue.get(timeout=240)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    merged = {}
    for part in gathered:
        assert not set(part) & set(merged)
        merged.update(part)
    single = _rows(range(world * PER_RANK))
    assert merged == single
    assert all(status == 0 for status, _ in single.values())


def test_reference_arm_under_torchrun_prints_one_line():
    """`bench.py --impl reference` launched as the benchmark contract launches
    N > 1 (torchrun, one process per rank): rank 0 alone times the oracle and
    prints one JSON line; the other rank exits 0 without work."""
    import json
    import subprocess
    import sys
    from conftest import ROOT
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["steps"] == 1 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0
