"""Helpers for the GPU parity tests: run the CUDA path through the C ABI and
bring results back as numpy."""
import numpy as np
import pytest
import torch

from paper_2609_16206_gb300 import workloads as W


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16206_gb300 import build
    build.build()
    from paper_2609_16206_gb300 import ctr
    ctr.lib()
    return ctr


def to_dev(trace_np: dict, dev="cuda") -> dict:
    """numpy rows [R, N] (or one row [N]) -> contiguous device tensors [R, N]."""
    out = {}
    for name, dt in (("arrival_us", np.int64), ("prompt_len", np.int32), ("true_out", np.int32),
                     ("pred_out", np.int32), ("slo_class", np.uint8)):
        a = np.ascontiguousarray(trace_np[name], dtype=dt)
        if a.ndim == 1:
            a = a[None, :]
        out[name] = torch.from_numpy(a).to(dev)
    return out


def gen(ctr, tc, n_replicas, n_req, offset=0):
    tr = ctr.empty_requests(n_replicas, n_req, "cuda")
    ctr.ctr_gen_trace(tc, n_replicas, offset, n_req, tr)
    torch.cuda.synchronize()
    return tr


def simulate(ctr, sc, sets, pols, tr, n_replicas, n_req, ws_bytes=None, routes=True):
    rows = n_replicas * len(sets) * len(pols)
    dev = "cuda"
    res = {"t_first_us": torch.full((rows, n_req), -7, dtype=torch.int64, device=dev),
           "t_done_us": torch.full((rows, n_req), -7, dtype=torch.int64, device=dev),
           "hash": torch.zeros(rows, dtype=torch.int64, device=dev),
           "status": torch.full((rows,), 99, dtype=torch.int32, device=dev)}
    if routes:
        res["i_pre"] = torch.full((rows, n_req), 255, dtype=torch.uint8, device=dev)
        res["i_dec"] = torch.full((rows, n_req), 255, dtype=torch.uint8, device=dev)
    if ws_bytes is None:
        ws = ctr.simulate_workspace(sc, rows, n_req, dev)
    else:
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    ctr.ctr_simulate(sc, sets, pols, tr, n_replicas, n_req, res["t_first_us"], res["t_done_us"], res["hash"],
                     res["status"], ws, i_pre=res.get("i_pre"), i_dec=res.get("i_dec"))
    torch.cuda.synchronize()
    out = {k: v.cpu().numpy() for k, v in res.items()}
    out["hash"] = out["hash"].astype(np.uint64)
    return out


def host_trace(tr: dict, r: int) -> dict:
    return {k: v[r].cpu().numpy() for k, v in tr.items()}
