"""CPU oracle for the marginal-cost routing simulation (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  It wraps
``ctr_oracle.c`` (plain single-threaded C, int64, fp64 scorer) with ctypes and numpy
and shares no code with the CUDA library: configurations arrive as plain
attribute objects (the workload presets) and are converted here into the
oracle's own C structs.

Functions follow the paper's sections as cited in ``ctr_oracle.c``:
Philox4x32-10 and the deterministic fp32 functions, the synthetic trace,
the event-heap simulator (sec. III-A cost, Algorithm 1, sec. III-D, sec. VI
batching, sec. IV-C baselines), SLO goodput / P99 TTFT, and the fp64
brute-force scorer.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ctr_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ENOMEM, EOVERFLOW, ETIMEOUT = 0, -1, -2, -3, -4


def build(force: bool = False) -> str:
    """Compile ctr_oracle.c into liboracle.so with gcc (no FMA contraction)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-Wall", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _TraceCfg(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("n_seeds", C.c_int64), ("arrival_kind", C.c_int64),
                ("rate_mreq", C.c_int64 * 2), ("dwell_mean_us", C.c_int64),
                ("prompt_mu", C.c_double), ("prompt_sigma", C.c_double),
                ("prompt_min", C.c_int64), ("prompt_max", C.c_int64),
                ("mix_short_thr", C.c_uint64),
                ("short_mu", C.c_double), ("short_sigma", C.c_double),
                ("long_mu", C.c_double), ("long_sigma", C.c_double),
                ("out_min", C.c_int64), ("out_max", C.c_int64),
                ("noise_sigma", C.c_double), ("pred_min", C.c_int64), ("pred_max", C.c_int64),
                ("n_classes", C.c_int64), ("class_thr", C.c_uint64 * 3)]


class _SimCfg(C.Structure):
    _fields_ = [("n_prefill", C.c_int64), ("n_decode", C.c_int64), ("kv_cap", C.c_int64),
                ("pre_base", C.c_int64), ("pre_per_tok", C.c_int64), ("xfer_per_tok", C.c_int64),
                ("dec_base", C.c_int64), ("dec_per_seq", C.c_int64), ("dec_kv_div", C.c_int64),
                ("n_classes", C.c_int64), ("ttft", C.c_int64 * 4), ("tpot", C.c_int64 * 4),
                ("max_steps", C.c_int64),
                ("cap_pending", C.c_int64), ("cap_waiting", C.c_int64), ("cap_active", C.c_int64),
                ("cap_prefill", C.c_int64), ("heur_thresh", C.c_int64), ("pre_batch_tokens", C.c_int64)]


class _Consts(C.Structure):
    _fields_ = [("tau_pre0", C.c_int64), ("tau_pre", C.c_int64), ("tau_dec", C.c_int64), ("w_q", C.c_int64),
                ("w_b_q8", C.c_int64), ("w_s_q8", C.c_int64), ("rho_q8", C.c_int64),
                ("sigma_q8", C.c_int64 * 4), ("ablate", C.c_int64),
                ("proxy_backlog", C.c_int64), ("poll_us", C.c_int64)]


class Stats(C.Structure):
    _fields_ = [("max_pending", C.c_int64), ("max_waiting", C.c_int64), ("max_active", C.c_int64),
                ("max_prefill", C.c_int64), ("max_reserved", C.c_int64), ("steps", C.c_int64),
                ("events", C.c_int64)]

    def as_dict(self):
        return {name: int(getattr(self, name)) for name, _ in self._fields_}


def _p(a, ctype):
    return a.ctypes.data_as(C.POINTER(ctype))


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = C.CDLL(_LIB_PATH)
            L.orc_philox4x32_10.argtypes = [C.POINTER(C.c_uint32), C.POINTER(C.c_uint32), C.POINTER(C.c_uint32)]
            for name in ("orc_det_logf_v", "orc_det_expf_v"):
                getattr(L, name).argtypes = [C.POINTER(C.c_float), C.POINTER(C.c_float), C.c_int64]
            for name in ("orc_det_ndtrif_v", "orc_unit_uniform_v"):
                getattr(L, name).argtypes = [C.POINTER(C.c_uint32), C.POINTER(C.c_float), C.c_int64]
            L.orc_gen_trace.argtypes = [C.POINTER(_TraceCfg), C.c_int64, C.c_int64, C.POINTER(C.c_int64),
                                        C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                        C.POINTER(C.c_uint8)]
            L.orc_simulate.argtypes = [C.POINTER(_SimCfg), C.POINTER(_Consts), C.c_int64, C.c_int64,
                                       C.POINTER(C.c_int64), C.POINTER(C.c_int32), C.POINTER(C.c_int32),
                                       C.POINTER(C.c_int32), C.POINTER(C.c_uint8), C.POINTER(C.c_uint8),
                                       C.POINTER(C.c_uint8), C.POINTER(C.c_int64), C.POINTER(C.c_int64),
                                       C.POINTER(C.c_int64), C.POINTER(C.c_int64), C.POINTER(C.c_uint64),
                                       C.POINTER(Stats)]
            L.orc_row_hash.restype = C.c_uint64
            L.orc_row_hash.argtypes = [C.c_int64, C.POINTER(C.c_uint8), C.POINTER(C.c_uint8),
                                       C.POINTER(C.c_int64), C.POINTER(C.c_int64)]
            L.orc_goodput.argtypes = [C.POINTER(_SimCfg), C.c_int64, C.POINTER(C.c_int64), C.POINTER(C.c_int32),
                                      C.POINTER(C.c_uint8), C.POINTER(C.c_int64), C.POINTER(C.c_int64),
                                      C.POINTER(C.c_int64), C.POINTER(C.c_int64)]
            L.orc_p99_tpot.argtypes = [C.c_int64, C.POINTER(C.c_int32), C.POINTER(C.c_int64), C.POINTER(C.c_int64),
                                       C.POINTER(C.c_int64)]
            L.orc_score_batch.argtypes = [C.POINTER(C.c_float), C.POINTER(C.c_float), C.POINTER(C.c_uint8),
                                          C.c_int64, C.POINTER(C.c_float), C.POINTER(C.c_float),
                                          C.POINTER(C.c_float), C.c_int64, C.POINTER(C.c_float),
                                          C.POINTER(C.c_int32), C.POINTER(C.c_double), C.POINTER(C.c_double)]
            L.orc_score_pairs.argtypes = [C.POINTER(C.c_float), C.POINTER(C.c_float), C.POINTER(C.c_uint8),
                                          C.POINTER(C.c_int64), C.POINTER(C.c_int64), C.c_int64,
                                          C.POINTER(C.c_float), C.POINTER(C.c_float), C.POINTER(C.c_float),
                                          C.POINTER(C.c_float), C.POINTER(C.c_double)]
            _lib = L
    return _lib


# ---------------------------------------------------------------- conversions
def _trace_cfg(tc) -> _TraceCfg:
    s = _TraceCfg()
    s.seed = int(tc.seed) & 0xFFFFFFFFFFFFFFFF
    s.n_seeds = int(tc.n_seeds)
    s.arrival_kind = int(tc.arrival_kind)
    s.rate_mreq[0], s.rate_mreq[1] = int(tc.rate_mreq[0]), int(tc.rate_mreq[1])
    s.dwell_mean_us = int(tc.dwell_mean_us)
    s.prompt_mu, s.prompt_sigma = float(tc.prompt_mu), float(tc.prompt_sigma)
    s.prompt_min, s.prompt_max = int(tc.prompt_min), int(tc.prompt_max)
    s.mix_short_thr = int(tc.mix_short_thr)
    s.short_mu, s.short_sigma = float(tc.short_mu), float(tc.short_sigma)
    s.long_mu, s.long_sigma = float(tc.long_mu), float(tc.long_sigma)
    s.out_min, s.out_max = int(tc.out_min), int(tc.out_max)
    s.noise_sigma = float(tc.noise_sigma)
    s.pred_min, s.pred_max = int(tc.pred_min), int(tc.pred_max)
    s.n_classes = int(tc.n_classes)
    thr = list(tc.class_thr) + [0] * (3 - len(tc.class_thr))
    for i in range(3):
        s.class_thr[i] = int(thr[i])
    return s


def _sim_cfg(sc) -> _SimCfg:
    s = _SimCfg()
    s.n_prefill, s.n_decode, s.kv_cap = int(sc.n_prefill), int(sc.n_decode), int(sc.kv_cap_tokens)
    s.pre_base, s.pre_per_tok, s.xfer_per_tok = int(sc.pre_base_us), int(sc.pre_us_per_tok), int(sc.xfer_us_per_tok)
    s.dec_base, s.dec_per_seq, s.dec_kv_div = int(sc.dec_base_us), int(sc.dec_us_per_seq), int(sc.dec_kv_tokens_per_us)
    s.n_classes = int(sc.n_classes)
    for i in range(4):
        s.ttft[i] = int(sc.ttft_slo_us[i]) if i < len(sc.ttft_slo_us) else 0
        s.tpot[i] = int(sc.tpot_slo_us[i]) if i < len(sc.tpot_slo_us) else 0
    s.max_steps = int(sc.max_steps_per_instance)
    s.cap_pending, s.cap_waiting = int(sc.cap_pending), int(sc.cap_waiting)
    s.cap_active, s.cap_prefill = int(sc.cap_active), int(sc.cap_prefill_ring)
    s.heur_thresh = int(sc.heuristic_threshold_tokens)
    s.pre_batch_tokens = int(getattr(sc, "prefill_batch_tokens", 0))
    return s


def _consts(cc) -> _Consts:
    s = _Consts()
    s.tau_pre0, s.tau_pre, s.tau_dec, s.w_q = int(cc.tau_pre0_us), int(cc.tau_pre_us), int(cc.tau_dec_us), int(cc.w_q_us)
    s.w_b_q8, s.w_s_q8, s.rho_q8 = int(cc.w_b_q8), int(cc.w_s_q8), int(cc.rho_q8)
    sig = list(cc.sigma_q8) + [256] * (4 - len(cc.sigma_q8))
    for i in range(4):
        s.sigma_q8[i] = int(sig[i])
    s.ablate = int(getattr(cc, "ablate", 0))
    s.proxy_backlog = int(getattr(cc, "proxy_backlog", 0))
    s.poll_us = int(getattr(cc, "poll_us", 0))
    return s


# ---------------------------------------------------------------- primitives
def philox4x32_10(ctr, key):
    c = np.asarray(ctr, dtype=np.uint32).copy()
    k = np.asarray(key, dtype=np.uint32).copy()
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_p(c, C.c_uint32), _p(k, C.c_uint32), _p(out, C.c_uint32))
    return out


def _vecf(name, x):
    x = np.ascontiguousarray(x, dtype=np.float32)
    y = np.empty_like(x)
    getattr(lib(), name)(_p(x, C.c_float), _p(y, C.c_float), x.size)
    return y


def _vecu(name, u):
    u = np.ascontiguousarray(u, dtype=np.uint32)
    y = np.empty(u.shape, np.float32)
    getattr(lib(), name)(_p(u, C.c_uint32), _p(y, C.c_float), u.size)
    return y


def det_logf(x):
    """fp32 natural log of the trace construction."""
    return _vecf("orc_det_logf_v", x)


def det_expf(x):
    """fp32 exp of the trace construction."""
    return _vecf("orc_det_expf_v", x)


def det_ndtrif(u):
    """fp32 normal quantile of the uniform (u + 1/2) 2^-32 of a 32-bit word."""
    return _vecu("orc_det_ndtrif_v", u)


def unit_uniform(u):
    """(u + 1/2) 2^-32 rounded once to fp32."""
    return _vecu("orc_unit_uniform_v", u)


# ---------------------------------------------------------------- trace
def gen_trace(tc, n_req: int, replica: int = 0) -> dict:
    """One replica's requests: arrival_us, prompt_len, true_out, pred_out, slo_class."""
    n = int(n_req)
    out = {"arrival_us": np.empty(n, np.int64), "prompt_len": np.empty(n, np.int32),
           "true_out": np.empty(n, np.int32), "pred_out": np.empty(n, np.int32),
           "slo_class": np.empty(n, np.uint8)}
    cfg = _trace_cfg(tc)
    rc = lib().orc_gen_trace(C.byref(cfg), int(replica), n, _p(out["arrival_us"], C.c_int64),
                             _p(out["prompt_len"], C.c_int32), _p(out["true_out"], C.c_int32),
                             _p(out["pred_out"], C.c_int32), _p(out["slo_class"], C.c_uint8))
    if rc != OK:
        raise ValueError(f"orc_gen_trace failed: {rc}")
    return out


def gen_traces(tc, n_replicas: int, n_req: int, replica_offset: int = 0) -> dict:
    """Rows [n_replicas, n_req] for replicas replica_offset .. + n_replicas - 1."""
    rows = [gen_trace(tc, n_req, replica_offset + r) for r in range(n_replicas)]
    return {key: np.stack([r[key] for r in rows]) if rows else np.empty((0, n_req)) for key in
            ("arrival_us", "prompt_len", "true_out", "pred_out", "slo_class")}


# ---------------------------------------------------------------- simulator
def simulate(sc, cc, policy: int, trace: dict) -> dict:
    """One row: returns per-request outputs, row hash, status and occupancy stats."""
    arr = np.ascontiguousarray(trace["arrival_us"], np.int64)
    p = np.ascontiguousarray(trace["prompt_len"], np.int32)
    o = np.ascontiguousarray(trace["true_out"], np.int32)
    oh = np.ascontiguousarray(trace["pred_out"], np.int32)
    cls = np.ascontiguousarray(trace["slo_class"], np.uint8)
    n = arr.size
    res = {"i_pre": np.zeros(n, np.uint8), "i_dec": np.zeros(n, np.uint8),
           "t_first_us": np.zeros(n, np.int64), "t_done_us": np.zeros(n, np.int64),
           "pre_end_us": np.zeros(n, np.int64), "t_ready_us": np.zeros(n, np.int64)}
    h = C.c_uint64(0)
    st = Stats()
    scfg, scc = _sim_cfg(sc), _consts(cc)
    rc = lib().orc_simulate(C.byref(scfg), C.byref(scc), int(policy), n, _p(arr, C.c_int64), _p(p, C.c_int32),
                            _p(o, C.c_int32), _p(oh, C.c_int32), _p(cls, C.c_uint8),
                            _p(res["i_pre"], C.c_uint8), _p(res["i_dec"], C.c_uint8),
                            _p(res["t_first_us"], C.c_int64), _p(res["t_done_us"], C.c_int64),
                            _p(res["pre_end_us"], C.c_int64), _p(res["t_ready_us"], C.c_int64),
                            C.byref(h), C.byref(st))
    res["status"] = int(rc)
    res["hash"] = int(h.value)
    res["stats"] = st.as_dict()
    return res


def row_hash(i_pre, i_dec, t_first, t_done) -> int:
    a = np.ascontiguousarray(i_pre, np.uint8)
    b = np.ascontiguousarray(i_dec, np.uint8)
    c = np.ascontiguousarray(t_first, np.int64)
    d = np.ascontiguousarray(t_done, np.int64)
    return int(lib().orc_row_hash(a.size, _p(a, C.c_uint8), _p(b, C.c_uint8), _p(c, C.c_int64), _p(d, C.c_int64)))


def goodput(sc, trace: dict, t_first, t_done):
    """(met_count, p99_ttft_us) of one row."""
    arr = np.ascontiguousarray(trace["arrival_us"], np.int64)
    o = np.ascontiguousarray(trace["true_out"], np.int32)
    cls = np.ascontiguousarray(trace["slo_class"], np.uint8)
    tf = np.ascontiguousarray(t_first, np.int64)
    td = np.ascontiguousarray(t_done, np.int64)
    met, p99 = C.c_int64(0), C.c_int64(0)
    scfg = _sim_cfg(sc)
    rc = lib().orc_goodput(C.byref(scfg), arr.size, _p(arr, C.c_int64), _p(o, C.c_int32), _p(cls, C.c_uint8),
                           _p(tf, C.c_int64), _p(td, C.c_int64), C.byref(met), C.byref(p99))
    if rc != OK:
        raise RuntimeError(f"orc_goodput failed: {rc}")
    return int(met.value), int(p99.value)


def p99_tpot(trace: dict, t_first, t_done) -> int:
    """Nearest-rank P99 of floor((t_done - t_first) / (o - 1)) over one row's requests with o >= 2 (-1: none)."""
    o = np.ascontiguousarray(trace["true_out"], np.int32)
    tf = np.ascontiguousarray(t_first, np.int64)
    td = np.ascontiguousarray(t_done, np.int64)
    out = C.c_int64(0)
    rc = lib().orc_p99_tpot(o.size, _p(o, C.c_int32), _p(tf, C.c_int64), _p(td, C.c_int64), C.byref(out))
    if rc != OK:
        raise RuntimeError(f"orc_p99_tpot failed: {rc}")
    return int(out.value)


# ---------------------------------------------------------------- scorer
def score_batch(p, oh, cls, Q, A, kap, consts):
    """fp64 brute force: (argmin int32, best fp64, second-best fp64) per request."""
    p = np.ascontiguousarray(p, np.float32)
    oh = np.ascontiguousarray(oh, np.float32)
    cls = np.ascontiguousarray(cls, np.uint8)
    Q = np.ascontiguousarray(Q, np.float32)
    A = np.ascontiguousarray(A, np.float32)
    kap = np.ascontiguousarray(kap, np.float32)
    cv = np.ascontiguousarray(consts, np.float32)
    n = p.size
    am = np.empty(n, np.int32)
    best = np.empty(n, np.float64)
    second = np.empty(n, np.float64)
    lib().orc_score_batch(_p(p, C.c_float), _p(oh, C.c_float), _p(cls, C.c_uint8), n, _p(Q, C.c_float),
                          _p(A, C.c_float), _p(kap, C.c_float), Q.size, _p(cv, C.c_float), _p(am, C.c_int32),
                          _p(best, C.c_double), _p(second, C.c_double))
    return am, best, second


def score_pairs(p, oh, cls, req_idx, inst_idx, Q, A, kap, consts):
    p = np.ascontiguousarray(p, np.float32)
    oh = np.ascontiguousarray(oh, np.float32)
    cls = np.ascontiguousarray(cls, np.uint8)
    ri = np.ascontiguousarray(req_idx, np.int64)
    di = np.ascontiguousarray(inst_idx, np.int64)
    Q = np.ascontiguousarray(Q, np.float32)
    A = np.ascontiguousarray(A, np.float32)
    kap = np.ascontiguousarray(kap, np.float32)
    cv = np.ascontiguousarray(consts, np.float32)
    out = np.empty(ri.size, np.float64)
    lib().orc_score_pairs(_p(p, C.c_float), _p(oh, C.c_float), _p(cls, C.c_uint8), _p(ri, C.c_int64),
                          _p(di, C.c_int64), ri.size, _p(Q, C.c_float), _p(A, C.c_float), _p(kap, C.c_float),
                          _p(cv, C.c_float), _p(out, C.c_double))
    return out
