"""Benchmark of the routing-simulation hot path on GB300.

One step = one pass of every hot-path row over one batch of synthetic input:
  - the bursty replica sweep (4,096 replicas x 20,000 requests, 2 prefill + 6
    decode instances, four policies): trace generation, simulation, goodput;
  - the standalone scorer (2^20 requests x 64 instances).
`value` is routed requests per second over the whole step (all ranks);
scored pairs per second and per-kernel times are reported beside it.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun each rank simulates its own 4,096 replicas (replica offset
rank * 4096; weak scaling, no collective on the data path).  --impl reference
times the CPU oracle (the only reference this method has) on the host cores.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import multiprocessing as mp
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_16206_gb300 import workloads as W  # noqa: E402

N_SCORE_REQ = 1 << 20
N_SCORE_INST = 64


# ---------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    def __init__(self, index: int):
        self.index = index
        self.samples = []
        self.proc = None
        self.thread = None

    def start(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.samples.append(parts)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = sorted(v for v in (num(s[1]) for s in self.samples) if v is not None)
        mx = [v for v in (num(s[2]) for s in self.samples) if v is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in self.samples for i in range(4) if s[5 + i].lower() == "active"})
        return {"sm_mhz": sm[len(sm) // 2] if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.samples)}


# ---------------------------------------------------------------- CPU oracle (baseline / reference arm)
def _oracle_replica(args):
    wl_name, replica, n_req, policies = args
    import oracle
    wl = {"replica_sweep": W.replica_sweep()}[wl_name]
    tr = oracle.gen_trace(wl.trace, n_req, replica=replica)
    routed = 0
    for pol in policies:
        res = oracle.simulate(wl.sim, W.CALIBRATED, pol, tr)
        oracle.goodput(wl.sim, tr, res["t_first_us"], res["t_done_us"])
        routed += n_req
    return routed


def oracle_rate(n_replicas: int, n_req: int, cores: int):
    """Routed requests per second of the oracle over a replica sample, one
    replica per process (spawned before any GPU work)."""
    import oracle
    oracle.build()
    tasks = [("replica_sweep", r, n_req, list(W.ALL_POLICIES)) for r in range(n_replicas)]
    ctx = mp.get_context("spawn")
    t0 = time.perf_counter()
    with ctx.Pool(processes=cores) as pool:
        routed = sum(pool.map(_oracle_replica, tasks, chunksize=1))
    dt = time.perf_counter() - t0
    return routed / dt, routed, dt


def sampled_parity(wl, offset, R, N, pols, tr, rstat, rhash, met, p99, score_in, score_state, sam, scost):
    """The benchmarked launch checked against the oracle on sampled rows,
    outside every timed region (the outputs of the last step: the timed
    steps and the end-to-end pass compute the same inputs).  The device trace
    of the first and last three replicas (all three seeds) must equal the
    oracle's bit for bit, every policy's row status and hash must equal the
    oracle simulation's, and so must the goodput count and P99 TTFT; 4,096
    sampled scorer requests must meet the scorer's bar (argmin identical
    outside the 1e-5 near-tie band, cost within 1e-6 relative)."""
    import numpy as np

    import oracle
    t0 = time.perf_counter()
    reps = sorted({0, 1, 2, R - 3, R - 2, R - 1} & set(range(R)))
    stat = rstat.cpu().numpy()
    hsh = rhash.cpu().numpy().astype(np.uint64)
    met_h, p99_h = met.cpu().numpy(), p99.cpu().numpy()
    bad, n_rows = [], 0
    for r in reps:
        ref = oracle.gen_trace(wl.trace, N, replica=offset + r)
        for key, v in ref.items():
            if not np.array_equal(tr[key][r].cpu().numpy(), v):
                bad.append(f"trace {key} replica {offset + r}")
        for j, pol in enumerate(pols):
            row = r * len(pols) + j
            n_rows += 1
            o = oracle.simulate(wl.sim, W.CALIBRATED, pol, ref)
            if int(stat[row]) != o["status"] or (o["status"] == 0 and int(hsh[row]) != o["hash"]):
                bad.append(f"row {row}")
            elif o["status"] == 0:
                if (int(met_h[row]), int(p99_h[row])) != oracle.goodput(wl.sim, ref, o["t_first_us"], o["t_done_us"]):
                    bad.append(f"goodput row {row}")
    p, oh, cls = score_in
    Q, A, kap = score_state
    idx = np.sort(np.random.default_rng(0).choice(p.size, 4096, replace=False))
    am, best, second = oracle.score_batch(p[idx], oh[idx], cls[idx], Q, A, kap, W.SCORE_CONSTS)
    am_d = sam.cpu().numpy()[idx]
    cost_d = scost.cpu().numpy()[idx].astype(np.float64)
    strict = (second - best) / best >= 1e-5
    chosen = oracle.score_pairs(p, oh, cls, idx, am_d, Q, A, kap, W.SCORE_CONSTS)
    score_ok = bool(np.array_equal(am_d[strict], am[strict]) and np.max(np.abs(cost_d - chosen) / chosen) <= 1e-6
                    and np.all(chosen <= best * (1 + 1e-5)))
    if not score_ok:
        bad.append("scorer")
    return {"ok": not bad, "rows": n_rows, "replicas": [offset + r for r in reps], "policies": len(pols),
            "checks": "trace rows bit-exact; row status + hash; goodput met + P99; scorer argmin + cost",
            "scorer_requests": int(idx.size), "mismatches": bad[:8],
            "seconds": round(time.perf_counter() - t0, 2)}


def run_reference(args, rank, world):
    if rank != 0:
        return 0
    cores = os.cpu_count() or 1
    wl = W.replica_sweep()
    n_rep = max(cores, 16)
    for _ in range(args.warmup and 1):
        oracle_rate(min(cores, 4), 2000, cores)
    vals, walls = [], []
    for _ in range(args.steps):
        v, routed, dt = oracle_rate(n_rep, wl.n_req, cores)
        vals.append(v)
        walls.append(dt)
    value = sum(vals) / len(vals)
    sample = f"{n_rep} replicas x {wl.n_req} requests x 4 policies per step (of 4,096 replicas)"
    line = {"impl": "reference", "metric": "routed requests/sec (replica sweep, 1 GB300)", "value": value,
            "unit": "routed requests/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000 * sum(walls) / len(walls), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": {"workload": wl.name, "replicas": wl.n_replicas, "requests_per_replica": wl.n_req,
                       "pool": "2P+6D", "policies": 4, "sample": sample},
            "cpu_baseline": {"value": value, "unit": "routed requests/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "routed requests/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- GPU arm
SIM_SOURCES = ("paper_2609_16206_gb300/csrc/sim.cu", "paper_2609_16206_gb300/csrc/ctr_internal.cuh", "include/ctr.h")
SCORE_SOURCES = ("paper_2609_16206_gb300/csrc/score.cu", "paper_2609_16206_gb300/csrc/ctr_internal.cuh", "include/ctr.h")


def _strip_comments(src: str) -> str:
    """C/C++ source without comments and trailing blanks (string and character
    literals kept), so that editing a comment does not change the key."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    return "\n".join(line.rstrip() for line in "".join(out).splitlines() if line.strip())


def _source_hash(sources=SIM_SOURCES) -> str:
    """Hash of the code (comments stripped) of the files that define a kernel (the simulator's by default)."""
    h = hashlib.sha256()
    for rel in sources:
        with open(os.path.join(ROOT, rel), encoding="utf-8") as f:
            h.update(rel.encode() + _strip_comments(f.read()).encode())
    return h.hexdigest()[:16]


def graph_ms(issue, stream, cap, reps):
    """Milliseconds per replay of a CUDA graph of the launches `issue(stream)`
    makes (captured on `cap`, replayed on `stream` after warm-up)."""
    import torch
    with torch.cuda.stream(stream):
        issue(stream)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    cap.wait_stream(stream)
    with torch.cuda.graph(graph, stream=cap):
        issue(cap)
    stream.wait_stream(cap)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(reps):
            graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    del graph
    return e0.elapsed_time(e1) / reps


def run_ours(args, rank, world, local_rank):
    import numpy as np
    import torch

    from paper_2609_16206_gb300 import build as ctr_build
    if rank == 0:
        ctr_build.build()
    if world > 1:
        torch.distributed.barrier()
    from paper_2609_16206_gb300 import ctr, sweep

    cpu_base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cores = os.cpu_count() or 1
        n_rep = max(2 * cores, 16)
        v, routed, dt = oracle_rate(n_rep, W.replica_sweep().n_req, cores)
        cpu_base = {"value": v, "unit": "routed requests/s", "cores": cores, "kind": "oracle",
                    "sample": f"{n_rep} replicas x 20000 requests x 4 policies, trace + simulation + goodput, "
                              f"one replica per process ({dt:.1f} s wall)"}

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    wl = W.replica_sweep(n_replicas=args.replicas or 4096, n_req=args.requests or 20_000)
    R, N = wl.n_replicas, wl.n_req
    pols = list(W.ALL_POLICIES)
    rows = R * len(pols)
    offset, _ = sweep.shard(rank, R)  # weak scaling: every rank its own block of replicas

    tr = ctr.empty_requests(R, N, dev)
    tf = torch.empty((rows, N), dtype=torch.int64, device=dev)
    td = torch.empty_like(tf)
    rhash = torch.empty(rows, dtype=torch.int64, device=dev)
    rstat = torch.empty(rows, dtype=torch.int32, device=dev)
    met = torch.empty(rows, dtype=torch.int64, device=dev)
    p99 = torch.empty(rows, dtype=torch.int64, device=dev)
    ws = ctr.simulate_workspace(wl.sim, rows, N, dev)
    p, oh, cls = W.score_requests(N_SCORE_REQ, seed=0)
    Q, A, kap = W.score_state(N_SCORE_INST, seed=1)
    sp, soh, scls = (torch.from_numpy(x).to(dev) for x in (p, oh, cls))
    sQ, sA, skap = (torch.from_numpy(x).to(dev) for x in (Q, A, kap))
    sam = torch.empty(N_SCORE_REQ, dtype=torch.int32, device=dev)
    scost = torch.empty(N_SCORE_REQ, dtype=torch.float32, device=dev)

    marks = {k: [] for k in ("gen", "sim", "score")}

    def step(timed: bool):
        """One pass of the hot path: trace generation, simulation (then each row's checksum and goodput in
        one pass over the outputs) and the scorer; with `timed`, CUDA events around each kernel, read after
        the timed region (no host synchronisation between steps)."""
        e = {k: [torch.cuda.Event(enable_timing=True) for _ in range(2)] for k in marks} if timed else None

        def mark(name, i):
            if timed:
                e[name][i].record(stream)
        mark("gen", 0)
        ctr.ctr_gen_trace(wl.trace, R, offset, N, tr, stream=stream)
        mark("gen", 1)
        mark("sim", 0)
        ctr.ctr_simulate(wl.sim, [W.CALIBRATED], pols, tr, R, N, tf, td, rhash, rstat, ws, met_count=met,
                         p99_ttft_us=p99, stream=stream)
        mark("sim", 1)
        mark("score", 0)
        ctr.ctr_score_batch(sp, soh, scls, sQ, sA, skap, W.SCORE_CONSTS, sam, scost, stream=stream)
        mark("score", 1)
        if timed:
            for k in e:
                marks[k].append(e[k])

    for _ in range(args.warmup):
        step(False)
    torch.cuda.synchronize()
    bad_rows = int((rstat != 0).sum())

    clocks = ClockSampler(local_rank)
    if rank == 0:
        clocks.start()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step(True)
    t1.record(stream)
    torch.cuda.synchronize()
    times = {k: sum(a.elapsed_time(z) for a, z in v) for k, v in marks.items()}
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop() if rank == 0 else None
    ms_total = t0.elapsed_time(t1)
    ms = torch.tensor([ms_total], dtype=torch.float64, device=dev)
    if world > 1:
        torch.distributed.all_reduce(ms, op=torch.distributed.ReduceOp.MAX)
    ms_total = float(ms.item())
    ms_step = ms_total / args.steps
    routed_per_step = rows * N * world
    value = routed_per_step / (ms_step / 1e3)
    per_kernel_ms = {k: v / args.steps for k, v in times.items()}

    # ---- end to end through the public API with host buffers (rank-local)
    host_tr = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in tr.items()}
    for k in tr:
        host_tr[k].copy_(tr[k])
    host_score = [torch.from_numpy(x).pin_memory() for x in (p, oh, cls)]
    out_host = {"met": torch.empty(rows, dtype=torch.int64, pin_memory=True),
                "p99": torch.empty(rows, dtype=torch.int64, pin_memory=True),
                "hash": torch.empty(rows, dtype=torch.int64, pin_memory=True),
                "status": torch.empty(rows, dtype=torch.int32, pin_memory=True),
                "am": torch.empty(N_SCORE_REQ, dtype=torch.int32, pin_memory=True),
                "cost": torch.empty(N_SCORE_REQ, dtype=torch.float32, pin_memory=True)}
    h2d = sum(v.numel() * v.element_size() for v in host_tr.values()) + sum(
        v.numel() * v.element_size() for v in host_score)
    d2h = sum(v.numel() * v.element_size() for v in out_host.values())

    # Double-buffered like a serving loop: step i + 1's inputs are copied from pinned host memory on a
    # second stream while step i computes; every step's inputs cross the link and its per-row results and
    # scorer outputs come back, all inside the timed region.
    bufs = [(dict(tr), (sp, soh, scls)),
            ({k: torch.empty_like(v) for k, v in tr.items()}, tuple(torch.empty_like(x) for x in (sp, soh, scls)))]
    copy_stream = torch.cuda.Stream(device=dev)
    ready = [torch.cuda.Event() for _ in range(2)]
    freed = [torch.cuda.Event() for _ in range(2)]
    for ev_ in freed:
        ev_.record(stream)

    def e2e_load(i):
        b = i % 2
        copy_stream.wait_event(freed[b])  # the compute that last read buffer b is done
        with torch.cuda.stream(copy_stream):
            for k in tr:
                bufs[b][0][k].copy_(host_tr[k], non_blocking=True)
            for d_, h_ in zip(bufs[b][1], host_score):
                d_.copy_(h_, non_blocking=True)
        ready[b].record(copy_stream)

    def e2e_compute(i):
        b = i % 2
        stream.wait_event(ready[b])
        t_, (p_, oh_, cls_) = bufs[b]
        ctr.ctr_simulate(wl.sim, [W.CALIBRATED], pols, t_, R, N, tf, td, rhash, rstat, ws, met_count=met,
                         p99_ttft_us=p99, stream=stream)
        ctr.ctr_score_batch(p_, oh_, cls_, sQ, sA, skap, W.SCORE_CONSTS, sam, scost, stream=stream)
        freed[b].record(stream)
        with torch.cuda.stream(stream):
            out_host["met"].copy_(met, non_blocking=True)
            out_host["p99"].copy_(p99, non_blocking=True)
            out_host["hash"].copy_(rhash, non_blocking=True)
            out_host["status"].copy_(rstat, non_blocking=True)
            out_host["am"].copy_(sam, non_blocking=True)
            out_host["cost"].copy_(scost, non_blocking=True)

    def e2e_run(n_steps):
        e2e_load(0)
        for i in range(n_steps):
            if i + 1 < n_steps:
                e2e_load(i + 1)
            e2e_compute(i)
        torch.cuda.synchronize()

    e2e_steps = max(3, args.steps)  # as many steps as the device-timed region
    if not args.no_e2e:
        e2e_run(2)
    if world > 1:
        torch.distributed.barrier()
    t_e0 = time.perf_counter()
    if not args.no_e2e:
        e2e_run(e2e_steps)
    e2e_s = (time.perf_counter() - t_e0) / e2e_steps
    e2e_t = torch.tensor([e2e_s], dtype=torch.float64, device=dev)
    if world > 1:
        torch.distributed.all_reduce(e2e_t, op=torch.distributed.ReduceOp.MAX)
    e2e_value = None if args.no_e2e else routed_per_step / float(e2e_t.item())

    # ---- the 2^20 scorer as its measurement rule asks: 30 buffer sets (534 MB, > 4x L2) launched back to
    # back from one CUDA graph, so every launch reads its inputs from HBM and launch gaps are not timed
    rot_sets = 30
    rot = [[torch.from_numpy(x).to(dev) for x in (p, oh, cls)] +
           [torch.empty(N_SCORE_REQ, dtype=torch.int32, device=dev),
            torch.empty(N_SCORE_REQ, dtype=torch.float32, device=dev)] for _ in range(rot_sets)]
    with torch.cuda.stream(stream):
        for b in rot:
            ctr.ctr_score_batch(b[0], b[1], b[2], sQ, sA, skap, W.SCORE_CONSTS, b[3], b[4], stream=stream)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream(device=dev)  # capture needs a stream of its own; replay runs on `stream`
    cap.wait_stream(stream)
    with torch.cuda.graph(graph, stream=cap):
        for b in rot:
            ctr.ctr_score_batch(b[0], b[1], b[2], sQ, sA, skap, W.SCORE_CONSTS, b[3], b[4], stream=cap)
    stream.wait_stream(cap)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    g_reps = 5
    g0 = torch.cuda.Event(enable_timing=True)
    g1 = torch.cuda.Event(enable_timing=True)
    g0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(g_reps):
            graph.replay()
    g1.record(stream)
    torch.cuda.synchronize()
    rot_ms = g0.elapsed_time(g1) / (g_reps * rot_sets)
    rot_ok = all(torch.equal(b[3], rot[0][3]) for b in rot[1:])
    del graph
    # the same harness around the scorer's traffic alone (ctr_score_stream_probe: its loads and stores on the
    # same grid, no arithmetic): the HBM throughput a kernel of this shape reaches at this size
    probe_ms = graph_ms(lambda st: [ctr.ctr_score_stream_probe(b[0], b[1], b[2], b[3], b[4], stream=st) for b in rot],
                        stream, cap, g_reps) / rot_sets
    del rot

    # ---- the scorer once more on 2^24 requests (285 MB per launch, beyond L2): its HBM roofline
    big_n = 1 << 24
    bp, boh, bcls = W.score_requests(big_n, seed=2)
    big = [[torch.from_numpy(x).to(dev) for x in (bp, boh, bcls)] +
           [torch.empty(big_n, dtype=torch.int32, device=dev), torch.empty(big_n, dtype=torch.float32, device=dev)]
           for _ in range(2)]  # two sets of 285 MB, alternated: each launch reads from HBM
    with torch.cuda.stream(stream):
        for b in big:
            ctr.ctr_score_batch(b[0], b[1], b[2], sQ, sA, skap, W.SCORE_CONSTS, b[3], b[4], stream=stream)
    torch.cuda.synchronize()
    reps = 10
    graph = torch.cuda.CUDAGraph()
    cap.wait_stream(stream)
    with torch.cuda.graph(graph, stream=cap):
        for i in range(reps):
            b = big[i % 2]
            ctr.ctr_score_batch(b[0], b[1], b[2], sQ, sA, skap, W.SCORE_CONSTS, b[3], b[4], stream=cap)
    stream.wait_stream(cap)
    with torch.cuda.stream(stream):
        graph.replay()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    big_ms = e0.elapsed_time(e1) / reps
    del graph
    big_probe_ms = graph_ms(lambda st: [ctr.ctr_score_stream_probe(b[0], b[1], b[2], b[3], b[4], stream=st)
                                        for b in (big[i % 2] for i in range(reps))], stream, cap, 1) / reps
    del big

    # ---- parity of the benchmarked launch itself, outside every timed region: the last step's trace,
    # row statuses and hashes, goodput counts and scorer outputs on sampled rows against the oracle
    parity = sampled_parity(wl, offset, R, N, pols, tr, rstat, rhash, met, p99, (p, oh, cls), (Q, A, kap), sam, scost) \
        if rank == 0 and not args.no_parity else None

    if rank != 0:
        return 0
    peaks = {}
    pk_path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(pk_path):
        with open(pk_path) as f:
            peaks = json.load(f)
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    issue_peak = n_sm * 4 * sm_max * 1e6 / 1e9   # G warp-instructions / s
    cnt = SIM_SLICE_COUNTERS.get(_source_hash())
    sim_roof = {"bound": "alu", "unit": "Gwarp-inst/s", "peak": issue_peak,
                "peak_source": f"{n_sm} SMs x 4 warp-inst/clk x {sm_max:.0f} MHz (max SM clock, "
                               + ("MEASURED_PEAKS.json)" if "sm_max_mhz" in peaks else "nominal)"),
                "achieved": None, "frac": None, "traffic": None,
                "inst_per_routed_request": None, "lane_efficiency": None, "dram_bytes_per_routed_request": None}
    if cnt is not None:
        # executed warp-instructions scale with routed requests (every row group's instruction stream is
        # fixed by its inputs), so the slice's count per routed request times this launch's routed requests
        # is this launch's count; DRAM bytes are scaled the same way (the slice holds fewer warps per SM)
        routed_launch = rows * N
        sim_roof["achieved"] = cnt["warp_inst_per_routed"] * routed_launch / (per_kernel_ms["sim"] / 1e3) / 1e9
        sim_roof["frac"] = sim_roof["achieved"] / issue_peak
        sim_roof["traffic"] = cnt["dram_bytes_per_routed"] * routed_launch
        sim_roof["inst_per_routed_request"] = cnt["warp_inst_per_routed"]
        sim_roof["lane_efficiency"] = cnt["thread_inst_per_warp_inst"] / 32
        sim_roof["dram_bytes_per_routed_request"] = cnt["dram_bytes_per_routed"]
        sim_roof["counters"] = cnt["slice"]
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    hbm_source = ("of measured (MEASURED_PEAKS.json hbm_gbs, a STREAM-style copy)" if "hbm_gbs" in peaks
                  else "of fallback (6.8 TB/s, an earlier GB300 copy measurement)")
    score_bytes = 17 * N_SCORE_REQ + 3 * 4 * N_SCORE_INST
    pairs_per_s = N_SCORE_REQ * N_SCORE_INST / (rot_ms / 1e3)  # graph-batched launches, inputs from HBM
    score_dram = SCORE_DRAM_PER_LAUNCH.get(_source_hash(SCORE_SOURCES))
    score_roof = {"bound": "hbm", "unit": "GB/s", "achieved": score_bytes / (rot_ms / 1e3) / 1e9,
                  "peak": hbm, "peak_source": hbm_source,
                  "traffic": None if score_dram is None else score_dram["read"] + score_dram["write"],
                  "launch_ms": rot_ms, "launch_ms_in_step": per_kernel_ms["score"],
                  "traffic_note": "no counters for this kernel source" if score_dram is None else
                  f"ncu DRAM read {score_dram['read'] / 1e6:.2f} MB, write {score_dram['write'] / 1e6:.2f} MB in "
                  "one launch of the step (the outputs are written back from L2 after it)",
                  "timing": f"{rot_sets} buffer sets ({rot_sets * score_bytes / 1e6:.0f} MB, > 4x L2) back to back "
                            f"from one CUDA graph, x{g_reps}; outputs identical across sets: {rot_ok}"}
    score_roof["frac"] = score_roof["achieved"] / hbm
    score_roof["ceiling_at_size"] = {
        "probe_launch_ms": probe_ms, "achieved": score_bytes / (probe_ms / 1e3) / 1e9,
        "frac_of_peak": score_bytes / (probe_ms / 1e3) / 1e9 / hbm, "scorer_frac_of_ceiling": probe_ms / rot_ms,
        "what": "ctr_score_stream_probe: the scorer's loads and stores alone (same grid, launch attributes and "
                "buffers, no arithmetic or envelope prologue), timed in the same graph"}
    big_bytes = 17 * big_n + 3 * 4 * N_SCORE_INST
    score_roof_big = {"bound": "hbm", "unit": "GB/s", "achieved": big_bytes / (big_ms / 1e3) / 1e9, "peak": hbm,
                      "peak_source": hbm_source,
                      "traffic": None, "launch_ms": big_ms, "requests": big_n}
    score_roof_big["frac"] = score_roof_big["achieved"] / hbm
    score_roof_big["ceiling_at_size"] = {
        "probe_launch_ms": big_probe_ms, "achieved": big_bytes / (big_probe_ms / 1e3) / 1e9,
        "frac_of_peak": big_bytes / (big_probe_ms / 1e3) / 1e9 / hbm, "scorer_frac_of_ceiling": big_probe_ms / big_ms}
    line = {
        "metric": "routed requests/sec (replica sweep, 1 GB300)", "value": value, "unit": "routed requests/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
        "data": "synthetic (seeded Philox traces shaped like the paper's mixed bursty workload)",
        "config": {"workload": wl.name, "replicas_per_gpu": R, "requests_per_replica": N, "pool": "2P+6D",
                   "policies": 4, "arrivals": "MMPP 3/12 req/s, 10 s mean dwell, seeds 0-2",
                   "score_workload": f"{N_SCORE_REQ} requests x {N_SCORE_INST} instances",
                   "l2": "inputs larger than L2 (1.7 GB trace, 5.2 GB of outputs per step)"},
        "scored_pairs_per_s": pairs_per_s,
        "kernel_ms": per_kernel_ms,
        "rows_failed": bad_rows,
        "roofline": sim_roof,
        "roofline_score": score_roof,
        "roofline_score_2p24": score_roof_big,
        "cpu_baseline": cpu_base,
        "parity_sampled": parity,
        "e2e": {"value": e2e_value, "unit": "routed requests/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "note": "per step: trace + scorer inputs copied in from pinned host memory (the next step's copy "
                         "overlaps this step's compute on a second stream, double-buffered), simulate + goodput + "
                         "score, per-row results and scorer outputs copied out; the host copy of the trace takes "
                         "the place of on-device trace generation (ctr_gen_trace), so this step does that much "
                         "less device work than the device-timed step; the first step's copy has no compute to "
                         "overlap (the pipeline fills once per run, which is timed over as many steps as the "
                         "device-timed region)",
                 "steps": e2e_steps},
        # per step: trace, simulation, the checksum's request-only mix table, checksum + goodput pass, scorer
        "gpu_launches": 5 * args.steps,
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    return 0


# Counters of one sim_kernel launch on a slice of the benchmarked workload
# (ncu sm__inst_executed.sum, smsp__thread_inst_executed.sum and DRAM bytes of
# 1,024 replicas x 20,000 requests x 4 policies, a few GB on the device),
# per routed request, keyed by a hash of the simulator's code: a stale entry
# (the kernel changed since the counters were taken) reports null.
SIM_SLICE_COUNTERS: dict = {
    "5b2cb8e0e1f5e9de": {"warp_inst_per_routed": 34162633267 / 81_920_000,
                         "thread_inst_per_warp_inst": 281165931678 / 34162633267,
                         "dram_bytes_per_routed": (2383411200 + 1563864576) / 81_920_000,
                         "slice": "ncu on one launch of 1,024 replicas x 20,000 requests x 4 policies "
                                  "(81.92 M routed requests): 3.416e10 warp-instructions, 2.812e11 thread-"
                                  "instructions, 2.383 GB DRAM read + 1.564 GB written"},
}

# DRAM bytes of one scorer launch (2^20 requests x 64 instances) inside the step.
SCORE_DRAM_PER_LAUNCH: dict = {
    "f16cba77579b1bc7": {"read": 9484800.0, "write": 0.0},
}


WORKLOADS = ("replica_sweep", "single_replica", "large_pool", "calibration_sweep", "document", "deployed_signals",
             "power_of_two", "noise_sweep")


def run_workload(args):
    """The other workload shapes (single GPU): trace generation, simulation under
    every policy and goodput per step, timed like the default workload; one
    JSON line.  For the record of their throughput beside the benchmarked
    sweep; the default run never takes this path."""
    import torch

    from paper_2609_16206_gb300 import build as ctr_build
    ctr_build.build()
    from paper_2609_16206_gb300 import ctr, sweep
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    name = args.workload
    info = {}
    if name == "noise_sweep":
        base = W.replica_sweep(n_req=args.requests or 20_000)
        seeds = args.replicas or 512
        n_sig = len(sweep.NOISE_SIGMAS)
        routed = n_sig * seeds * len(W.ALL_POLICIES) * base.n_req
        cfg = {"workload": f"noise_sweep_2p6d_{n_sig}x{seeds}x{base.n_req}", "noise_sigmas": list(sweep.NOISE_SIGMAS),
               "replicas": n_sig * seeds, "requests_per_replica": base.n_req, "policies": len(W.ALL_POLICIES)}
        state = {}

        def step():
            state["out"] = sweep.noise_sweep(base, seeds=seeds)
    elif name == "calibration_sweep":
        t_sat = time.perf_counter()
        sat = sweep.calibration_saturation()
        torch.cuda.synchronize()
        info["saturation_search_s"] = time.perf_counter() - t_sat
        n_sets = len(W.mispriced_sets())
        routed = 5 * 4 * 4 * 16 * (n_sets + 3) * 10_000
        cfg = {"workload": "calibration_sweep_2p3d-2p7d_256seeds_x10000", "widths": "3-7 decode (2P)",
               "replicas_per_width": 256, "learned_sets": n_sets, "baselines": 3,
               "loads": "0.8 / 0.967 / 1.133 / 1.3 x saturation", "mixes": "100/83/67/50 % short"}
        state = {}

        def step():
            state["out"] = sweep.calibration_sweep(sat)
    else:
        if name == "single_replica":
            wl = W.single_replica()
        elif name == "document":
            wl = W.document(n_replicas=args.replicas or 4096, n_req=args.requests or 10_000)
        elif name in ("deployed_signals", "power_of_two"):
            wl = W.replica_sweep(n_replicas=args.replicas or 4096, n_req=args.requests or 20_000)
            if name == "deployed_signals":
                wl = dataclasses.replace(wl, name=wl.name + "_deployed", consts=[W.as_deployed(W.CALIBRATED)])
            else:
                wl = dataclasses.replace(wl, name=wl.name + "_p2",
                                         policies=(W.POLICY_LEARNED_P2, W.POLICY_RR, W.POLICY_JSQ, W.POLICY_HEURISTIC))
        elif name == "large_pool":
            base = W.large_pool(n_replicas=args.replicas or 16384, n_req=args.requests or 50_000)
            t_sat = time.perf_counter()
            sat = sweep.saturation_rate([base.trace], base.sim, n_req=10_000)[0]
            info["saturation_search_s"] = time.perf_counter() - t_sat
            info["rate_mreq"] = sweep.load_rate(sat, 1.2)
            wl = dataclasses.replace(base, trace=base.trace.replace(rate_mreq=(info["rate_mreq"],) * 2))
        else:
            wl = W.replica_sweep(n_replicas=args.replicas or 4096, n_req=args.requests or 20_000)
        pols = list(wl.policies)
        rows = wl.n_replicas * len(wl.consts) * len(pols)
        routed = rows * wl.n_req
        buf = sweep.alloc(wl.sim, wl.n_replicas, rows, wl.n_req, dev)
        cfg = {"workload": wl.name, "replicas": wl.n_replicas, "requests_per_replica": wl.n_req,
               "pool": f"{wl.sim.n_prefill}P+{wl.sim.n_decode}D", "policies": len(pols),
               "prefill_batch_tokens": wl.sim.prefill_batch_tokens}

        def step():
            sweep.run_step(wl.trace, wl.sim, wl.consts, pols, wl.n_replicas, wl.n_req, 0, buf, stream=stream)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    clocks = ClockSampler(0)
    clocks.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step()
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms_step = t0.elapsed_time(t1) / args.steps
    if name == "calibration_sweep":
        failed = sum(int((b.row_status != 0).sum()) for pair in state["out"].values() for b in pair)
    elif name == "noise_sweep":
        failed = int((state["out"][0].row_status != 0).sum())
    else:
        failed = int((buf.row_status != 0).sum())
    cfg.update(info)
    print(json.dumps({
        "metric": "routed requests/sec", "value": routed / (ms_step / 1e3), "unit": "routed requests/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "dtype": "int64", "data": "synthetic", "config": cfg,
        "rows_failed": failed, "note": "trace generation + simulation + goodput per step", "clocks": clk}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end pass")
    ap.add_argument("--no-parity", action="store_true", help="skip the sampled oracle check of the benchmarked launch")
    ap.add_argument("--replicas", type=int, default=None,
                    help="replicas per GPU (profiling a smaller case; default: the benchmarked 4,096)")
    ap.add_argument("--requests", type=int, default=None, help="requests per replica (default 20,000)")
    ap.add_argument("--workload", choices=WORKLOADS, default="replica_sweep",
                    help="another workload shape, timed alone on one GPU (default: the benchmarked sweep)")
    args = ap.parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.workload != "replica_sweep":
        if world > 1:
            raise SystemExit("--workload other than replica_sweep runs on one GPU")
        return run_workload(args)
    if world > 1:
        import torch
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
    try:
        return run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
