"""Workload presets and seeded input generators.

This module holds parameter values and seeded numpy draws only -- none of the
method's arithmetic.  It is shared by the CUDA binding's callers (tests,
bench) and by the CPU oracle's callers, which convert these plain objects
into their own structures.

The presets are the synthetic stand-ins for the paper's workloads: the
paper measures on a vLLM/NIXL testbed (sec. IV-A) and publishes no traces, so
request lengths follow the length profiles of Table 1 as lognormal laws and
arrivals are Poisson or a two-state Markov-modulated Poisson process (the
"mixed bursty" family).  Times are integer microseconds.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import numpy as np

# natural logs, correctly rounded to fp64 (hex so every machine parses the same value)
LN_16 = float.fromhex("0x1.62e42fefa39efp+1")
LN_128 = float.fromhex("0x1.3687a9f1af2b1p+2")
LN_512 = float.fromhex("0x1.8f40b5ed9812dp+2")
LN_1024 = float.fromhex("0x1.bb9d3beb8c86bp+2")
LN_2048 = float.fromhex("0x1.e7f9c1e980fa9p+2")

POLICY_LEARNED, POLICY_RR, POLICY_JSQ, POLICY_HEURISTIC, POLICY_LEARNED_P2 = 0, 1, 2, 3, 4
POLICY_NAMES = {POLICY_LEARNED: "learned", POLICY_RR: "round_robin", POLICY_JSQ: "least_loaded",
                POLICY_HEURISTIC: "length_heuristic", POLICY_LEARNED_P2: "learned_power_of_two"}
ABLATE_PREDICTED_LENGTH, ABLATE_PRESSURE, ABLATE_SLO = 1, 2, 4
PROXY_POLL_US = 50_000               # the deployed proxy's occupancy poll period (sec. IV-A)
ALL_POLICIES = (POLICY_LEARNED, POLICY_RR, POLICY_JSQ, POLICY_HEURISTIC)


def prob_to_u32_threshold(prob: float) -> int:
    """floor(prob * 2^32 + 1/2): a uniform 32-bit word u is below it w.p. ~prob."""
    return int(np.floor(prob * 4294967296.0 + 0.5))


@dataclass
class TraceCfg:
    """Synthetic request trace (one Philox key per replica seed)."""
    seed: int = 0
    n_seeds: int = 1                 # replica g uses seed + (g mod n_seeds), sub-stream g // n_seeds
    arrival_kind: int = 0            # 0 Poisson, 1 two-state MMPP starting in the low state
    rate_mreq: tuple = (4000, 4000)  # milli-requests per second (low, high)
    dwell_mean_us: int = 10_000_000
    prompt_mu: float = LN_512
    prompt_sigma: float = 1.0
    prompt_min: int = 16
    prompt_max: int = 8192
    mix_short_thr: int = prob_to_u32_threshold(0.7)
    short_mu: float = LN_128
    short_sigma: float = 0.8
    long_mu: float = LN_1024
    long_sigma: float = 0.6
    out_min: int = 1
    out_max: int = 4096
    noise_sigma: float = 0.3
    pred_min: int = 1
    pred_max: int = 1 << 17
    n_classes: int = 2
    class_thr: tuple = (prob_to_u32_threshold(0.6),)

    def replace(self, **kw) -> "TraceCfg":
        return dataclasses.replace(self, **kw)


@dataclass
class SimCfg:
    """Cluster physics, SLO classes and structure capacities of one pool shape."""
    n_prefill: int = 1
    n_decode: int = 3
    kv_cap_tokens: int = 200_000
    pre_base_us: int = 20_000
    pre_us_per_tok: int = 150
    xfer_us_per_tok: int = 20
    dec_base_us: int = 15_000
    dec_us_per_seq: int = 200
    dec_kv_tokens_per_us: int = 1000      # 1 ns per resident KV token, floored
    n_classes: int = 2
    ttft_slo_us: tuple = (1_000_000, 5_000_000)
    tpot_slo_us: tuple = (100_000, 250_000)
    max_steps_per_instance: int = (1 << 31) - (1 << 21)  # the largest budget the library accepts
    cap_pending: int = 1024
    cap_waiting: int = 1024
    cap_active: int = 1024
    cap_prefill_ring: int = 1024
    heuristic_threshold_tokens: int = 512
    prefill_batch_tokens: int = 0         # 0: serial FCFS prefill; > 0: batched prefill, token budget per batch

    def replace(self, **kw) -> "SimCfg":
        return dataclasses.replace(self, **kw)


@dataclass
class CostConsts:
    """Fixed-point cost constants of the learned router (weights x256)."""
    tau_pre0_us: int = 20_000
    tau_pre_us: int = 150
    tau_dec_us: int = 15_200
    w_q_us: int = 5_000
    w_b_q8: int = 256
    w_s_q8: int = 256
    rho_q8: int = 256
    sigma_q8: tuple = (512, 256, 256, 256)
    ablate: int = 0                  # ABLATE_* bits: features replaced by their neutral value
    proxy_backlog: int = 0           # 1: backlog from the proxy's priced in-flight ledger, 0: true remaining work
    poll_us: int = 0                 # > 0: KV occupancy polled every poll_us (the proxy's 50 ms); 0: live

    def replace(self, **kw) -> "CostConsts":
        return dataclasses.replace(self, **kw)


CALIBRATED = CostConsts()


@dataclass
class SweepWorkload:
    name: str
    trace: TraceCfg
    sim: SimCfg
    consts: list = field(default_factory=lambda: [CALIBRATED])
    policies: tuple = ALL_POLICIES
    n_replicas: int = 1
    n_req: int = 2000


def single_replica() -> SweepWorkload:
    """1 prefill + 3 decode, 2,000 requests, Poisson 4 req/s, two SLO classes."""
    return SweepWorkload("single_replica_1p3d_2000req", TraceCfg(), SimCfg(), n_replicas=1, n_req=2000)


def replica_sweep(n_replicas: int = 4096, n_req: int = 20_000) -> SweepWorkload:
    """2 prefill + 6 decode, MMPP 3 / 12 req/s with 10 s mean dwell, seeds 0,1,2."""
    tc = TraceCfg(seed=0, n_seeds=3, arrival_kind=1, rate_mreq=(3000, 12000), dwell_mean_us=10_000_000)
    sc = SimCfg(n_prefill=2, n_decode=6)
    return SweepWorkload(f"replica_sweep_2p6d_{n_replicas}x{n_req}_mmpp", tc, sc,
                         n_replicas=n_replicas, n_req=n_req)


U32_ALL = 1 << 32                    # a threshold every 32-bit word is below
PREFILL_BATCH_TOKENS = 8192          # token budget of one prefill batch in the batched-prefill presets


def chat(n_replicas: int = 256, n_req: int = 10_000, rate_mreq: int = 9_000) -> SweepWorkload:
    """Table 1 'chat' (short in, short out): the single-replica prompt law, every
    output from the short component; 2P+6D, Poisson."""
    tc = TraceCfg(rate_mreq=(rate_mreq, rate_mreq), mix_short_thr=U32_ALL)
    return SweepWorkload(f"chat_2p6d_{n_replicas}x{n_req}", tc, SimCfg(n_prefill=2, n_decode=6),
                         n_replicas=n_replicas, n_req=n_req)


def reasoning(n_replicas: int = 256, n_req: int = 10_000, rate_mreq: int = 4_000) -> SweepWorkload:
    """Table 1 'reasoning' (short in, long out): every output from the long component."""
    tc = TraceCfg(rate_mreq=(rate_mreq, rate_mreq), mix_short_thr=0)
    return SweepWorkload(f"reasoning_2p6d_{n_replicas}x{n_req}", tc, SimCfg(n_prefill=2, n_decode=6),
                         n_replicas=n_replicas, n_req=n_req)


def document(n_replicas: int = 256, n_req: int = 10_000, rate_mreq: int = 5_000,
             batch_tokens: int = PREFILL_BATCH_TOKENS) -> SweepWorkload:
    """Table 1 'document' (up to 4k in, short out; stresses prefill compute and
    KV transfer): prompts lognormal around 2,048 tokens clipped to [16, 4096],
    outputs from the short component, 2P+6D, Poisson, batched prefill with a
    `batch_tokens` budget (0 = serial prefill)."""
    tc = TraceCfg(rate_mreq=(rate_mreq, rate_mreq), prompt_mu=LN_2048, prompt_sigma=0.5, prompt_max=4096,
                  mix_short_thr=U32_ALL)
    sc = SimCfg(n_prefill=2, n_decode=6, prefill_batch_tokens=batch_tokens)
    return SweepWorkload(f"document_2p6d_{n_replicas}x{n_req}", tc, sc, n_replicas=n_replicas, n_req=n_req)


def large_pool(n_replicas: int = 16384, n_req: int = 50_000, rate_mreq: int = 33_000) -> SweepWorkload:
    """4 prefill + 28 decode, C = 100,000, three SLO classes 30/40/30, predictor noise 0.6."""
    tc = TraceCfg(rate_mreq=(rate_mreq, rate_mreq), noise_sigma=0.6, n_classes=3,
                  class_thr=(prob_to_u32_threshold(0.3), prob_to_u32_threshold(0.7)))
    sc = SimCfg(n_prefill=4, n_decode=28, kv_cap_tokens=100_000, n_classes=3,
                ttft_slo_us=(500_000, 2_000_000, 10_000_000), tpot_slo_us=(50_000, 150_000, 300_000),
                cap_pending=4096, cap_waiting=4096, cap_active=1024, cap_prefill_ring=16384)
    cc = CostConsts(sigma_q8=(512, 384, 256, 256))
    return SweepWorkload(f"large_pool_4p28d_{n_replicas}x{n_req}", tc, sc, consts=[cc],
                         n_replicas=n_replicas, n_req=n_req)


def as_deployed(cc: CostConsts) -> CostConsts:
    """The same constants with the deployed proxy's signals: ledger backlog and a 50 ms occupancy poll."""
    return cc.replace(proxy_backlog=1, poll_us=PROXY_POLL_US)


def mispriced_sets(base: CostConsts = CALIBRATED, factors=(0.5, 0.75, 1.5, 2.0)) -> list:
    """The calibrated set followed by the 4^3 grid of (tau_pre0, tau_pre, tau_dec)
    scalings, each scaled value rounded half up."""
    def sc(v, f):
        return int(np.floor(v * f + 0.5))
    out = [base]
    for a in factors:
        for b in factors:
            for c in factors:
                out.append(base.replace(tau_pre0_us=sc(base.tau_pre0_us, a), tau_pre_us=sc(base.tau_pre_us, b),
                                        tau_dec_us=sc(base.tau_dec_us, c)))
    return out


# ---------------------------------------------------------------- standalone scorer inputs
SCORE_N_CONST = 13
SCORE_CONSTS = np.array([
    1.0,        # w_b
    1.0,        # w_s
    0.005,      # w_q, seconds per active sequence
    1.0,        # rho
    0.020,      # tau_pre0, s
    0.00015,    # tau_pre, s / prompt token
    0.0152,     # tau_dec, s / output token
    0.020,      # tau_act, s of committed work per active decode sequence
    1.0 / 200_000.0,  # 1 / KV capacity
    2.0, 1.0, 1.0, 1.0,  # sigma per SLO class
], dtype=np.float32)


def score_requests(n_req: int, seed: int = 0):
    """(prompt_len, pred_out, slo_class) drawn from the single-replica laws with numpy."""
    rng = np.random.default_rng(seed)
    p = np.clip(np.floor(np.exp(LN_512 + rng.standard_normal(n_req)) + 0.5), 16, 8192)
    short = rng.random(n_req) < 0.7
    z = rng.standard_normal(n_req)
    o = np.clip(np.floor(np.exp(np.where(short, LN_128 + 0.8 * z, LN_1024 + 0.6 * z)) + 0.5), 1, 4096)
    oh = np.clip(np.floor(o * np.exp(0.3 * rng.standard_normal(n_req)) + 0.5), 1, 1 << 17)
    cls = (rng.random(n_req) >= 0.6).astype(np.uint8)
    return p.astype(np.float32), oh.astype(np.float32), cls


def score_state(n_inst: int, seed: int = 1):
    """(queued prefill tokens, active decode sequences, KV occupancy) per instance."""
    rng = np.random.default_rng(seed)
    Q = rng.integers(0, 65536, size=n_inst, endpoint=True).astype(np.float32)
    A = rng.integers(0, 256, size=n_inst, endpoint=True).astype(np.float32)
    kap = rng.random(n_inst, dtype=np.float32)
    return Q, A, kap
