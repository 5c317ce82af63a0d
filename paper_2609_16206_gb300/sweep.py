"""Host-side orchestration of replica sweeps over the C ABI.

* ``shard`` / ``shard_split`` -- which replicas a rank owns (weak and strong
  scaling); replicas are independent, so ranks exchange nothing.
* ``SweepBuffers`` / ``run_step`` -- device buffers and one pass of the hot
  path for a workload: trace generation, simulation under every policy and
  constant set, goodput.
* ``saturation_rate`` -- the arrival rate at which round-robin goodput
  crosses 1/2 (sec. IV-B runs each workload at the load where round-robin is
  half-way into collapse, located by probing): an integer bisection over
  milli-requests per second, every probe a GPU simulation.
* ``calibration_sweep_cfgs`` / ``load_rate`` -- the mispriced-constants x
  pool-width sweep grid and its offered rates.
* ``noise_sweep`` -- the predictor-noise sweep of sec. V-G: the same replicas
  at every noise level (common random numbers), one simulation call.
* ``policy_table`` -- Table 2's columns per policy (goodput, P99 TTFT, P99
  TPOT), each the mean over a workload's replicas (the paper averages its
  rows over arrival traces).
* ``resumable_sweep`` / ``read_journal`` -- a sweep in replica chunks with a
  per-chunk journal, so that a killed sweep restarts where it stopped (the
  paper journals every run per request and resumes it, sec. IV-B); every row
  depends on its seeds alone, so a resumed sweep equals an uninterrupted one.

Everything here is argument marshalling and control flow; the arithmetic runs
in the CUDA kernels behind ``ctr``.
"""
from __future__ import annotations

import dataclasses
import hashlib
import json
import os

import numpy as np
import torch

from . import ctr
from . import workloads as W


def shard(rank: int, replicas_per_rank: int) -> tuple:
    """Weak scaling: rank r simulates replicas [r * n, (r + 1) * n)."""
    return rank * replicas_per_rank, replicas_per_rank


def shard_split(total: int, world: int, rank: int) -> tuple:
    """Strong scaling: a contiguous, near-equal split of `total` replicas."""
    base, extra = divmod(total, world)
    count = base + (1 if rank < extra else 0)
    offset = rank * base + min(rank, extra)
    return offset, count


@dataclasses.dataclass
class SweepBuffers:
    trace: dict
    t_first: torch.Tensor
    t_done: torch.Tensor
    row_hash: torch.Tensor
    row_status: torch.Tensor
    met: torch.Tensor
    p99: torch.Tensor
    workspace: torch.Tensor


def alloc(sim_cfg, n_replicas: int, n_rows: int, n_req: int, device) -> SweepBuffers:
    return SweepBuffers(
        trace=ctr.empty_requests(n_replicas, n_req, device),
        t_first=torch.empty((n_rows, n_req), dtype=torch.int64, device=device),
        t_done=torch.empty((n_rows, n_req), dtype=torch.int64, device=device),
        row_hash=torch.empty(n_rows, dtype=torch.int64, device=device),
        row_status=torch.empty(n_rows, dtype=torch.int32, device=device),
        met=torch.empty(n_rows, dtype=torch.int64, device=device),
        p99=torch.empty(n_rows, dtype=torch.int64, device=device),
        workspace=ctr.simulate_workspace(sim_cfg, n_rows, n_req, device))


def run_step(trace_cfg, sim_cfg, const_sets, policies, n_replicas: int, n_req: int, replica_offset: int,
             buf: SweepBuffers, stream=None, gen: bool = True):
    """Trace generation (unless gen is False), then simulation with each row's
    goodput computed in the pass that completes its checksum; rows are
    (replica, set, policy) row-major."""
    if gen:
        ctr.ctr_gen_trace(trace_cfg, n_replicas, replica_offset, n_req, buf.trace, stream=stream)
    ctr.ctr_simulate(sim_cfg, const_sets, policies, buf.trace, n_replicas, n_req, buf.t_first, buf.t_done,
                     buf.row_hash, buf.row_status, buf.workspace, met_count=buf.met, p99_ttft_us=buf.p99,
                     stream=stream)


def saturation_rate(trace_cfgs, sim_cfg, n_req: int = 10_000, lo: int = 1, hi: int = 200_000, steps: int = 24,
                    device="cuda") -> list:
    """For every trace law in `trace_cfgs` (arrival_kind / rate replaced by a
    Poisson rate), the largest rate in milli-requests/s found by a `steps`-step
    integer bisection on [lo, hi] at which the round-robin goodput of one
    replica (seed of the law, replica 0) is at least 1/2.  All laws are probed
    together, one simulation call per step."""
    k = len(trace_cfgs)
    lows = [lo] * k
    highs = [hi] * k
    buf = alloc(sim_cfg, k, k, n_req, device)
    for _ in range(steps):
        mids = [(a + b) // 2 for a, b in zip(lows, highs)]
        for i, (tc, mid) in enumerate(zip(trace_cfgs, mids)):
            law = tc.replace(arrival_kind=0, rate_mreq=(max(mid, 1), max(mid, 1)))
            view = {name: t[i:i + 1] for name, t in buf.trace.items()}
            ctr.ctr_gen_trace(law, 1, 0, n_req, view)
        run_step(None, sim_cfg, [W.CALIBRATED], [W.POLICY_RR], k, n_req, 0, buf, gen=False)
        met = buf.met.cpu().tolist()
        status = buf.row_status.cpu().tolist()
        for i in range(k):
            ok = status[i] == ctr.CTR_OK and 2 * met[i] >= n_req
            if ok:
                lows[i] = mids[i]
            else:
                highs[i] = mids[i]
    return lows


def calibration_sweep_cfgs(widths=(3, 4, 5, 6, 7), mixes=(1.0, 5 / 6, 2 / 3, 1 / 2),
                           loads=(0.8, 29 / 30, 17 / 15, 1.3), seeds: int = 16):
    """The pool-width x trace-mix x load grid of the mispriced-constants sweep:
    per width, per (mix, load), `seeds` replicas (distinct sub-streams of seed 0).
    Returns [(width, mix, load, trace_cfg_without_rate)]."""
    out = []
    for w in widths:
        for mix in mixes:
            for load in loads:
                tc = W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(mix), seed=0, n_seeds=1)
                out.append((w, mix, load, tc))
    return out


def load_rate(sat_mreq: int, load: float) -> int:
    """Offered rate = load x saturation rate, rounded half up, at least 1."""
    return max(1, int(sat_mreq * load + 0.5))


NOISE_SIGMAS = (0.0, 0.25, 0.5, 0.75, 1.0, 1.25, 1.5)  # sec. V-G injects up to 150 % relative error


def noise_sweep(wl, sigmas=NOISE_SIGMAS, seeds: int = 16, const_sets=None, policies=None, device="cuda"):
    """Every predictor-noise level in `sigmas` on the same `seeds` replicas of
    workload `wl` (replica slice [i * seeds, (i + 1) * seeds) has noise
    sigmas[i]; arrivals, lengths and the noise draws are shared, only the
    prediction's spread changes), simulated and scored in one call each.
    Returns (buffers, n_replicas)."""
    const_sets = const_sets or wl.consts
    policies = policies or list(W.ALL_POLICIES)
    R = len(sigmas) * seeds
    rows = R * len(const_sets) * len(policies)
    buf = alloc(wl.sim, R, rows, wl.n_req, device)
    for i, sg in enumerate(sigmas):
        view = {name: t[i * seeds:(i + 1) * seeds] for name, t in buf.trace.items()}
        ctr.ctr_gen_trace(wl.trace.replace(noise_sigma=float(sg)), seeds, 0, wl.n_req, view)
    run_step(None, wl.sim, const_sets, policies, R, wl.n_req, 0, buf, gen=False)
    return buf, R


def calibration_sweep(sat_rates, widths=(3, 4, 5, 6, 7), mixes=(1.0, 5 / 6, 2 / 3, 1 / 2),
                      loads=(0.8, 29 / 30, 17 / 15, 1.3), seeds: int = 16, n_req: int = 10_000,
                      const_sets=None, device="cuda"):
    """The mispriced-constants x pool-width sweep (sec. V-B, the calibration
    study), batched: per pool width one trace buffer holds every (mix, load,
    seed) replica -- replica (i * len(loads) + j) * seeds + s has mix i, load
    j and sub-stream s -- and two simulation calls cover it: the learned
    router under every constant set, and the three baselines under the
    calibrated set.  `sat_rates[w][i]` is the saturation rate (milli-requests
    per second) of width w and mix i; the offered rate is load x that.
    Returns {width: (learned SweepBuffers, baseline SweepBuffers)}."""
    const_sets = const_sets or W.mispriced_sets()
    base_pols = [W.POLICY_RR, W.POLICY_JSQ, W.POLICY_HEURISTIC]
    out = {}
    for w in widths:
        sc = W.SimCfg(n_prefill=2, n_decode=w)
        R = len(mixes) * len(loads) * seeds
        learned = alloc(sc, R, R * len(const_sets), n_req, device)
        base = alloc(sc, R, R * len(base_pols), n_req, device)
        for i, mix in enumerate(mixes):
            for j, load in enumerate(loads):
                rate = load_rate(sat_rates[w][i], load)
                tc = W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(mix), rate_mreq=(rate, rate))
                lo = (i * len(loads) + j) * seeds
                view = {name: t[lo:lo + seeds] for name, t in learned.trace.items()}
                ctr.ctr_gen_trace(tc, seeds, 0, n_req, view)
        base.trace = learned.trace
        run_step(None, sc, const_sets, [W.POLICY_LEARNED], R, n_req, 0, learned, gen=False)
        run_step(None, sc, [W.CALIBRATED], base_pols, R, n_req, 0, base, gen=False)
        learned.workspace = base.workspace = None  # released once the launches complete
        out[w] = (learned, base)
    return out


def calibration_saturation(widths=(3, 4, 5, 6, 7), mixes=(1.0, 5 / 6, 2 / 3, 1 / 2), n_req: int = 10_000,
                           device="cuda") -> dict:
    """Saturation rate per (width, mix) for `calibration_sweep`."""
    laws = [W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(m)) for m in mixes]
    return {w: saturation_rate(laws, W.SimCfg(n_prefill=2, n_decode=w), n_req=n_req, device=device)
            for w in widths}


def policy_table(wl, n_replicas: int = None, n_req: int = None, policies=None, const_set=None,
                 device="cuda") -> dict:
    """{policy name: {"goodput", "p99_ttft_s", "p99_tpot_s", "rows_failed"}}: Table 2's columns for one
    workload, each the mean over its replicas of the per-row values (goodput = met / requests; the P99s in
    seconds, rows without a multi-token request left out of the TPOT mean).  One trace, one simulation of
    every policy, one goodput pass with P99 TPOT."""
    R = n_replicas or wl.n_replicas
    N = n_req or wl.n_req
    pols = list(policies or wl.policies)
    cc = const_set or wl.consts[0]
    buf = alloc(wl.sim, R, R * len(pols), N, device)
    run_step(wl.trace, wl.sim, [cc], pols, R, N, 0, buf)
    tpot = torch.empty(R * len(pols), dtype=torch.int64, device=device)
    ctr.ctr_goodput(wl.sim, buf.trace, R, len(pols), N, buf.t_first, buf.t_done, buf.met, buf.p99,
                    p99_tpot_us=tpot)
    torch.cuda.synchronize()
    ok = (buf.row_status == ctr.CTR_OK).view(R, len(pols))
    met = buf.met.view(R, len(pols)).double()
    p99 = buf.p99.view(R, len(pols)).double()
    tp = tpot.view(R, len(pols)).double()
    out = {}
    for j, pol in enumerate(pols):
        good = ok[:, j]
        has_tpot = good & (tp[:, j] >= 0)
        out[W.POLICY_NAMES[pol]] = {
            "goodput": float((met[good, j] / max(N, 1)).mean()) if good.any() else None,
            "p99_ttft_s": float(p99[good, j].mean() / 1e6) if good.any() else None,
            "p99_tpot_s": float(tp[has_tpot, j].mean() / 1e6) if has_tpot.any() else None,
            "rows_failed": int((~good).sum()),
        }
    return out


# ---------------------------------------------------------------- resumable sweeps
JOURNAL_VERSION = 1
_U64 = (1 << 64) - 1
RESULT_FIELDS = ("row_hash", "row_status", "met", "p99_ttft_us")


def sweep_fingerprint(wl, const_sets, policies, chunk: int) -> str:
    """A digest of everything that determines a sweep's rows and chunking (a journal of another sweep is refused)."""
    d = {"version": JOURNAL_VERSION, "trace": dataclasses.asdict(wl.trace), "sim": dataclasses.asdict(wl.sim),
         "consts": [dataclasses.asdict(c) for c in const_sets], "policies": [int(p) for p in policies],
         "n_replicas": int(wl.n_replicas), "n_req": int(wl.n_req), "chunk": int(chunk)}
    return hashlib.sha256(json.dumps(d, sort_keys=True).encode()).hexdigest()


def read_journal(path: str, fingerprint: str, repair: bool = False) -> dict:
    """{replica offset: record} of the chunks in a journal (one JSON line per finished chunk).  A last line
    without its newline is an append that was cut short: it is ignored (and, with repair, cut off the file so
    the next append starts on a line of its own).  Any other unreadable line, or a line of another sweep,
    raises ValueError."""
    done = {}
    if not os.path.exists(path):
        return done
    with open(path, "rb") as f:
        data = f.read()
    good_end, pos = 0, 0
    while pos < len(data):
        nl = data.find(b"\n", pos)
        if nl < 0:  # the torn tail of an interrupted append
            break
        line = data[pos:nl]
        pos = nl + 1
        if line.strip():
            try:
                rec = json.loads(line)
            except json.JSONDecodeError as e:
                raise ValueError(f"{path}: unreadable journal line ending at byte {nl}") from e
            if rec.get("fingerprint") != fingerprint:
                raise ValueError(f"{path} is the journal of another sweep")
            done[int(rec["offset"])] = rec
        good_end = pos
    if repair and good_end < len(data):
        with open(path, "r+b") as f:
            f.truncate(good_end)
    return done


def _gpu_chunk_runner(wl, const_sets, policies, chunk: int, device):
    """run(offset, count): trace, simulation and goodput of replicas [offset, offset + count) on the GPU."""
    per = len(const_sets) * len(policies)
    buf = alloc(wl.sim, chunk, chunk * per, wl.n_req, device)

    def run(off: int, cnt: int) -> dict:
        rows = cnt * per
        trace = {k: v[:cnt] for k, v in buf.trace.items()}
        ctr.ctr_gen_trace(wl.trace, cnt, off, wl.n_req, trace)
        ctr.ctr_simulate(wl.sim, const_sets, policies, trace, cnt, wl.n_req, buf.t_first[:rows], buf.t_done[:rows],
                         buf.row_hash[:rows], buf.row_status[:rows], buf.workspace, met_count=buf.met[:rows],
                         p99_ttft_us=buf.p99[:rows])
        torch.cuda.synchronize()
        return {"row_hash": [int(x) & _U64 for x in buf.row_hash[:rows].tolist()],
                "row_status": buf.row_status[:rows].tolist(), "met": buf.met[:rows].tolist(),
                "p99_ttft_us": buf.p99[:rows].tolist()}
    return run


def resumable_sweep(wl, journal: str, chunk: int = 256, const_sets=None, policies=None, device="cuda",
                    max_chunks: int = None, run_chunk=None):
    """The rows of workload `wl` (replica x constant set x policy) simulated in chunks of `chunk` replicas.
    Each finished chunk's per-row checksum, status, met count and P99 TTFT go to `journal` as one JSON line,
    flushed and fsynced, before the next chunk starts; chunks already in the journal are not simulated again.
    So a sweep that is killed (a lost rank, a pre-empted job) restarts where it stopped, and its rows equal
    those of one uninterrupted run: a row is a function of its replica's seeds alone.  `max_chunks` stops
    after that many new chunks.  Returns {field: numpy array over all rows, replica-major} once every chunk
    is journaled, else None.  `run_chunk(offset, count) -> {field: list}` replaces the GPU runner (tests)."""
    const_sets = list(const_sets or wl.consts)
    policies = list(policies or wl.policies)
    if chunk < 1:
        raise ValueError("chunk must be positive")
    fp = sweep_fingerprint(wl, const_sets, policies, chunk)
    done = read_journal(journal, fp, repair=True)
    offsets = list(range(0, wl.n_replicas, chunk))
    todo = [o for o in offsets if o not in done]
    if max_chunks is not None:
        todo = todo[:max_chunks]
    if todo:
        run = run_chunk or _gpu_chunk_runner(wl, const_sets, policies, chunk, device)
        for off in todo:
            cnt = min(chunk, wl.n_replicas - off)
            rec = {"fingerprint": fp, "offset": off, "count": cnt}
            rec.update(run(off, cnt))
            with open(journal, "a") as f:
                f.write(json.dumps(rec) + "\n")
                f.flush()
                os.fsync(f.fileno())
            done[off] = rec
    if any(o not in done for o in offsets):
        return None
    out = {}
    for k in RESULT_FIELDS:
        dt = np.uint64 if k == "row_hash" else np.int64
        out[k] = np.concatenate([np.zeros(0, dt)] + [np.asarray(done[o][k], dtype=dt) for o in offsets])
    return out
