"""ctypes binding of libctr.so (include/ctr.h).

Argument marshalling only: configurations (the dataclasses of ``workloads``)
become the C structs of ``ctr.h``; torch tensors become device pointers; the
current torch stream is passed as ``cudaStream_t``.  Every step of the
computation runs in the CUDA kernels of ``csrc/``.  There is no fallback: if
``libctr.so`` is missing or CUDA is unavailable the calls raise.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libctr.so")
# the bounds-checked build of the same library (build.build(checked=True)); use_library() switches to it
LIB_CHECKED_PATH = os.path.join(_HERE, "libctr_checked.so")

CTR_OK, CTR_EINVAL, CTR_ECUDA, CTR_EOVERFLOW, CTR_ETIMEOUT, CTR_EBOUNDS = 0, -1, -2, -3, -4, -5
CTR_MAX_INSTANCES = 32
CTR_MAX_CONST_SETS = 128
CTR_MAX_REQUESTS = 1 << 23
CTR_MAX_STEPS_PER_INSTANCE = (1 << 31) - (1 << 21)
CTR_SCORE_N_CONST = 13
CTR_SCORE_MAX_INST = 256
CTR_SCORE_MAX_REQ = 1 << 40
CTR_WS_SIMULATE = 0

REQUEST_FIELDS = (("arrival_us", torch.int64), ("prompt_len", torch.int32), ("true_out", torch.int32),
                  ("pred_out", torch.int32), ("slo_class", torch.uint8))


class CtrError(RuntimeError):
    def __init__(self, func, code, detail=None):
        self.code = code
        super().__init__(f"{func} failed: {code} ({detail if detail is not None else ctr_strerror(code)})")


# ---------------------------------------------------------------- C structs (ctr.h)
class CtrRequests(C.Structure):
    _fields_ = [("arrival_us", C.c_void_p), ("prompt_len", C.c_void_p), ("true_out", C.c_void_p),
                ("pred_out", C.c_void_p), ("slo_class", C.c_void_p)]


class CtrTraceCfg(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("n_seeds", C.c_int32), ("arrival_kind", C.c_int32),
                ("rate_mreq", C.c_int64 * 2), ("dwell_mean_us", C.c_int64),
                ("prompt_mu", C.c_double), ("prompt_sigma", C.c_double),
                ("prompt_min", C.c_int32), ("prompt_max", C.c_int32), ("mix_short_thr", C.c_uint64),
                ("short_mu", C.c_double), ("short_sigma", C.c_double), ("long_mu", C.c_double),
                ("long_sigma", C.c_double), ("out_min", C.c_int32), ("out_max", C.c_int32),
                ("noise_sigma", C.c_double), ("pred_min", C.c_int32), ("pred_max", C.c_int32),
                ("n_classes", C.c_int32), ("reserved0", C.c_int32), ("class_thr", C.c_uint64 * 3)]


class CtrSimCfg(C.Structure):
    _fields_ = [("n_prefill", C.c_int32), ("n_decode", C.c_int32), ("kv_cap_tokens", C.c_int64),
                ("pre_base_us", C.c_int64), ("pre_us_per_tok", C.c_int64), ("xfer_us_per_tok", C.c_int64),
                ("dec_base_us", C.c_int64), ("dec_us_per_seq", C.c_int64), ("dec_kv_tokens_per_us", C.c_int64),
                ("n_classes", C.c_int32), ("heuristic_threshold_tokens", C.c_int32),
                ("ttft_slo_us", C.c_int64 * 4), ("tpot_slo_us", C.c_int64 * 4),
                ("max_steps_per_instance", C.c_int64),
                ("cap_pending", C.c_int32), ("cap_waiting", C.c_int32), ("cap_active", C.c_int32),
                ("cap_prefill_ring", C.c_int32), ("prefill_batch_tokens", C.c_int64)]


class CtrCostConsts(C.Structure):
    _fields_ = [("tau_pre0_us", C.c_int64), ("tau_pre_us", C.c_int64), ("tau_dec_us", C.c_int64),
                ("w_q_us", C.c_int64), ("w_b_q8", C.c_int32), ("w_s_q8", C.c_int32), ("rho_q8", C.c_int32),
                ("sigma_q8", C.c_int32 * 4), ("ablate", C.c_uint32),
                ("backlog_signal", C.c_uint32), ("occupancy_poll_us", C.c_int64)]


_lock = threading.RLock()
_lib = None


def lib():
    """The loaded libctr.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                msg = f"{LIB_PATH} is missing: build it with paper_2609_16206_gb300/build.py"
                raise CtrError("load", CTR_ECUDA, detail=msg) from FileNotFoundError(msg)
            L = C.CDLL(LIB_PATH)
            vp, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
            L.ctr_gen_trace.argtypes = [C.POINTER(CtrTraceCfg), i32, i64, i64, CtrRequests, vp]
            L.ctr_gen_trace.restype = C.c_int
            L.ctr_score_batch.argtypes = [vp, vp, vp, i64, vp, vp, vp, i32, C.POINTER(C.c_float), vp, vp, vp, vp]
            L.ctr_score_batch.restype = C.c_int
            L.ctr_score_stream_probe.argtypes = [vp, vp, vp, i64, vp, vp, vp]
            L.ctr_score_stream_probe.restype = C.c_int
            L.ctr_workspace_bytes.argtypes = [i32, C.POINTER(CtrSimCfg), i64, i64]
            L.ctr_workspace_bytes.restype = C.c_size_t
            L.ctr_simulate.argtypes = [C.POINTER(CtrSimCfg), C.POINTER(CtrCostConsts), i32, C.POINTER(i32), i32,
                                       CtrRequests, i32, i64, vp, vp, vp, vp, vp, vp, vp, vp, vp, C.c_size_t, vp]
            L.ctr_simulate.restype = C.c_int
            L.ctr_simulate_noalloc.argtypes = [C.POINTER(CtrSimCfg), C.POINTER(CtrCostConsts), i32, C.POINTER(i32),
                                               i32, CtrRequests, i32, i64, vp, vp, vp, vp, vp, vp, vp]
            L.ctr_simulate_noalloc.restype = C.c_int
            L.ctr_goodput.argtypes = [C.POINTER(CtrSimCfg), CtrRequests, i32, i32, i64, vp, vp, vp, vp, vp, vp]
            L.ctr_goodput.restype = C.c_int
            L.ctr_strerror.argtypes = [C.c_int]
            L.ctr_strerror.restype = C.c_char_p
            L.ctr_abi_version.restype = C.c_int
            L.ctr_bounds_checked.restype = C.c_int
            _lib = L
    return _lib


def use_library(path: str) -> str:
    """Make every following call go to the library at `path` (LIB_PATH or
    LIB_CHECKED_PATH); returns the path in use before."""
    global _lib, LIB_PATH
    with _lock:
        before = LIB_PATH
        LIB_PATH = path
        _lib = None
        lib()
    return before


def ctr_strerror(code: int) -> str:
    if _lib is None and not os.path.exists(LIB_PATH):
        return "libctr.so not loaded"
    try:
        return lib().ctr_strerror(int(code)).decode()
    except (CtrError, OSError):
        return "libctr.so not loaded"


def _check(func: str, rc: int):
    if rc != CTR_OK:
        raise CtrError(func, rc)


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


# ---------------------------------------------------------------- struct conversion
def trace_cfg_struct(tc) -> CtrTraceCfg:
    s = CtrTraceCfg()
    s.seed = int(tc.seed) & 0xFFFFFFFFFFFFFFFF
    s.n_seeds, s.arrival_kind = int(tc.n_seeds), int(tc.arrival_kind)
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


def sim_cfg_struct(sc) -> CtrSimCfg:
    s = CtrSimCfg()
    s.n_prefill, s.n_decode = int(sc.n_prefill), int(sc.n_decode)
    s.kv_cap_tokens = int(sc.kv_cap_tokens)
    s.pre_base_us, s.pre_us_per_tok, s.xfer_us_per_tok = int(sc.pre_base_us), int(sc.pre_us_per_tok), int(sc.xfer_us_per_tok)
    s.dec_base_us, s.dec_us_per_seq = int(sc.dec_base_us), int(sc.dec_us_per_seq)
    s.dec_kv_tokens_per_us = int(sc.dec_kv_tokens_per_us)
    s.n_classes, s.heuristic_threshold_tokens = int(sc.n_classes), int(sc.heuristic_threshold_tokens)
    for i in range(4):
        s.ttft_slo_us[i] = int(sc.ttft_slo_us[i]) if i < len(sc.ttft_slo_us) else 0
        s.tpot_slo_us[i] = int(sc.tpot_slo_us[i]) if i < len(sc.tpot_slo_us) else 0
    s.max_steps_per_instance = int(sc.max_steps_per_instance)
    s.cap_pending, s.cap_waiting = int(sc.cap_pending), int(sc.cap_waiting)
    s.cap_active, s.cap_prefill_ring = int(sc.cap_active), int(sc.cap_prefill_ring)
    s.prefill_batch_tokens = int(getattr(sc, "prefill_batch_tokens", 0))
    return s


def consts_array(sets):
    arr = (CtrCostConsts * len(sets))()
    for i, cc in enumerate(sets):
        a = arr[i]
        a.tau_pre0_us, a.tau_pre_us, a.tau_dec_us, a.w_q_us = (int(cc.tau_pre0_us), int(cc.tau_pre_us),
                                                                int(cc.tau_dec_us), int(cc.w_q_us))
        a.w_b_q8, a.w_s_q8, a.rho_q8 = int(cc.w_b_q8), int(cc.w_s_q8), int(cc.rho_q8)
        sig = list(cc.sigma_q8) + [256] * (4 - len(cc.sigma_q8))
        for c in range(4):
            a.sigma_q8[c] = int(sig[c])
        a.ablate = int(getattr(cc, "ablate", 0))
        a.backlog_signal = int(getattr(cc, "proxy_backlog", 0))
        a.occupancy_poll_us = int(getattr(cc, "poll_us", 0))
    return arr


def requests_struct(req: dict) -> CtrRequests:
    r = CtrRequests()
    for name, dtype in REQUEST_FIELDS:
        t = req[name]
        if t.dtype != dtype:
            raise ValueError(f"{name} must be {dtype}")
        setattr(r, name, _ptr(t))
    return r


# ---------------------------------------------------------------- allocation helpers (torch plumbing)
def empty_requests(n_replicas: int, n_req: int, device="cuda") -> dict:
    return {name: torch.empty((n_replicas, n_req), dtype=dt, device=device) for name, dt in REQUEST_FIELDS}


def simulate_workspace(sim_cfg, n_rows: int, n_req: int, device="cuda") -> torch.Tensor:
    n = ctr_workspace_bytes(CTR_WS_SIMULATE, sim_cfg, n_rows, n_req)
    if n == 0:
        raise CtrError("ctr_workspace_bytes", CTR_EINVAL)
    return torch.empty(n, dtype=torch.uint8, device=device)


# ---------------------------------------------------------------- the ABI
def ctr_gen_trace(trace_cfg, n_replicas: int, replica_offset: int, n_req: int, out: dict, stream=None):
    cfg = trace_cfg_struct(trace_cfg)
    _check("ctr_gen_trace", lib().ctr_gen_trace(C.byref(cfg), int(n_replicas), int(replica_offset), int(n_req),
                                                requests_struct(out), _stream(stream)))


def ctr_score_batch(prompt_len, pred_out, slo_class, q_tokens, n_active, kv_occ, consts, out_argmin, out_cost,
                    status=None, stream=None):
    cv = (C.c_float * CTR_SCORE_N_CONST)(*[float(x) for x in consts])
    _check("ctr_score_batch", lib().ctr_score_batch(
        _ptr(prompt_len), _ptr(pred_out), _ptr(slo_class), int(prompt_len.numel()), _ptr(q_tokens), _ptr(n_active),
        _ptr(kv_occ), int(q_tokens.numel()), cv, _ptr(out_argmin), _ptr(out_cost), _ptr(status), _stream(stream)))


def ctr_score_stream_probe(prompt_len, pred_out, slo_class, out_argmin, out_cost, stream=None):
    """The scorer's memory traffic alone (a measurement aid; see include/ctr.h)."""
    _check("ctr_score_stream_probe", lib().ctr_score_stream_probe(
        _ptr(prompt_len), _ptr(pred_out), _ptr(slo_class), int(prompt_len.numel()), _ptr(out_argmin),
        _ptr(out_cost), _stream(stream)))


def ctr_workspace_bytes(which: int, sim_cfg, n_rows: int, n_req: int) -> int:
    cfg = sim_cfg_struct(sim_cfg)
    return int(lib().ctr_workspace_bytes(int(which), C.byref(cfg), int(n_rows), int(n_req)))


def ctr_simulate(sim_cfg, const_sets, policies, trace: dict, n_replicas: int, n_req: int, t_first_us, t_done_us,
                 row_hash, row_status, workspace, i_pre=None, i_dec=None, met_count=None, p99_ttft_us=None,
                 stream=None):
    cfg = sim_cfg_struct(sim_cfg)
    sets = consts_array(list(const_sets))
    pols = (C.c_int32 * len(policies))(*[int(p) for p in policies])
    _check("ctr_simulate", lib().ctr_simulate(
        C.byref(cfg), sets, len(sets), pols, len(policies), requests_struct(trace), int(n_replicas), int(n_req),
        _ptr(i_pre), _ptr(i_dec), _ptr(t_first_us), _ptr(t_done_us), _ptr(row_hash), _ptr(row_status),
        _ptr(met_count), _ptr(p99_ttft_us), _ptr(workspace), int(workspace.numel() * workspace.element_size()),
        _stream(stream)))


def ctr_simulate_noalloc(sim_cfg, const_sets, policies, trace: dict, n_replicas: int, n_req: int, t_first_us,
                         t_done_us, row_hash, row_status, i_pre=None, i_dec=None, stream=None):
    """ctr_simulate without a workspace: the library's fixed scratch array is
    used instead, for callers that cannot allocate device memory."""
    cfg = sim_cfg_struct(sim_cfg)
    sets = consts_array(list(const_sets))
    pols = (C.c_int32 * len(policies))(*[int(p) for p in policies])
    _check("ctr_simulate_noalloc", lib().ctr_simulate_noalloc(
        C.byref(cfg), sets, len(sets), pols, len(policies), requests_struct(trace), int(n_replicas), int(n_req),
        _ptr(i_pre), _ptr(i_dec), _ptr(t_first_us), _ptr(t_done_us), _ptr(row_hash), _ptr(row_status),
        _stream(stream)))


def ctr_goodput(sim_cfg, trace: dict, n_replicas: int, rows_per_replica: int, n_req: int, t_first_us, t_done_us,
                met_count, p99_ttft_us, p99_tpot_us=None, stream=None):
    cfg = sim_cfg_struct(sim_cfg)
    _check("ctr_goodput", lib().ctr_goodput(
        C.byref(cfg), requests_struct(trace), int(n_replicas), int(rows_per_replica), int(n_req), _ptr(t_first_us),
        _ptr(t_done_us), _ptr(met_count), _ptr(p99_ttft_us), _ptr(p99_tpot_us), _stream(stream)))


def ctr_abi_version() -> int:
    return int(lib().ctr_abi_version())


def ctr_bounds_checked() -> int:
    return int(lib().ctr_bounds_checked())
