"""The C ABI library (no GPU needed): it loads, exports every function that
include/ctr.h declares, its ctypes binding lays structs out exactly as the
header does, and the product path refuses to run without CUDA."""
import ctypes
import os
import re
import subprocess

import pytest

from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "ctr.h")


@pytest.fixture(scope="module")
def libctr():
    from paper_2609_16206_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(ctr_\w+)\s*\(", text, flags=re.M)))


def test_exports_every_declared_function(libctr):
    names = declared_functions()
    assert {"ctr_gen_trace", "ctr_score_batch", "ctr_simulate", "ctr_goodput"} <= set(names)
    for name in names:
        assert hasattr(libctr, name), name


def test_static_entry_points_run_without_gpu(libctr):
    libctr.ctr_strerror.restype = ctypes.c_char_p
    assert libctr.ctr_strerror(-3).decode().startswith("a fixed-capacity")
    assert libctr.ctr_strerror(-5).decode().startswith("an index fell outside")
    assert libctr.ctr_abi_version() == 8
    assert libctr.ctr_bounds_checked() == 0


def test_bounds_checked_library_exports_the_same_entry_points():
    """libctr_checked.so (the simulator compiled with CTR_BOUNDS_CHECK=1) is the
    same ABI: every declared function, the same version, and it says it is the
    checked build."""
    from paper_2609_16206_gb300 import build
    L = ctypes.CDLL(build.build(checked=True))
    for name in declared_functions():
        assert hasattr(L, name), name
    assert L.ctr_abi_version() == 8
    assert L.ctr_bounds_checked() == 1


def test_step_budget_bound_checked_on_the_host():
    """max_steps_per_instance is accepted up to CTR_MAX_STEPS_PER_INSTANCE (the
    kernel's step counters are 32-bit) and rejected above it, before any device
    work (zero rows)."""
    from paper_2609_16206_gb300 import ctr
    from paper_2609_16206_gb300 import workloads as W
    L = ctr.lib()
    sets = ctr.consts_array([W.CALIBRATED])
    pols = (ctypes.c_int32 * 1)(0)

    def call(steps):
        cfg = ctr.sim_cfg_struct(W.SimCfg(max_steps_per_instance=steps))
        return L.ctr_simulate(ctypes.byref(cfg), sets, 1, pols, 1, ctr.CtrRequests(), 0, 0, None, None, None, None,
                              None, None, None, None, None, 0, None)
    assert W.SimCfg().max_steps_per_instance == ctr.CTR_MAX_STEPS_PER_INSTANCE == (1 << 31) - (1 << 21)
    assert call(ctr.CTR_MAX_STEPS_PER_INSTANCE) == ctr.CTR_OK
    assert call(1) == ctr.CTR_OK
    assert call(ctr.CTR_MAX_STEPS_PER_INSTANCE + 1) == ctr.CTR_EINVAL
    assert call(0) == ctr.CTR_EINVAL


def test_request_count_bound_checked_on_the_host():
    """CTR_MAX_REQUESTS requests per replica (the 23-bit request index of the
    packed heap keys) is accepted and one more is rejected, by every entry
    that takes a request count, before any device work."""
    from paper_2609_16206_gb300 import ctr
    from paper_2609_16206_gb300 import workloads as W
    L = ctr.lib()
    M = ctr.CTR_MAX_REQUESTS
    assert M == 1 << 23
    cfg = ctr.sim_cfg_struct(W.SimCfg())
    sets = ctr.consts_array([W.CALIBRATED])
    pols = (ctypes.c_int32 * 1)(0)

    def sim(n_req):  # zero replicas: validation only
        return L.ctr_simulate(ctypes.byref(cfg), sets, 1, pols, 1, ctr.CtrRequests(), 0, n_req, None, None, None,
                              None, None, None, None, None, None, 0, None)

    def goodput(n_req):
        return L.ctr_goodput(ctypes.byref(cfg), ctr.CtrRequests(), 0, 4, n_req, None, None, None, None, None, None)
    assert sim(M) == ctr.CTR_OK and sim(M + 1) == ctr.CTR_EINVAL and sim(-1) == ctr.CTR_EINVAL
    assert goodput(M) == ctr.CTR_OK and goodput(M + 1) == ctr.CTR_EINVAL
    tcfg = ctr.trace_cfg_struct(W.TraceCfg())
    assert L.ctr_gen_trace(ctypes.byref(tcfg), 1, 0, M + 1, ctr.CtrRequests(), None) == ctr.CTR_EINVAL
    # the standalone scorer and its traffic probe: at most CTR_SCORE_MAX_REQ requests
    S = ctr.CTR_SCORE_MAX_REQ
    assert S == 1 << 40
    cv = (ctypes.c_float * ctr.CTR_SCORE_N_CONST)(*W.SCORE_CONSTS)
    buf = ctypes.create_string_buffer(64)
    ptr = ctypes.cast(ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 16, ctypes.c_void_p)
    for n in (S + 4, (1 << 63) - 4):
        assert L.ctr_score_batch(ptr, ptr, ptr, n, ptr, ptr, ptr, 4, cv, ptr, ptr, None, None) == ctr.CTR_EINVAL
        assert L.ctr_score_stream_probe(ptr, ptr, ptr, n, ptr, ptr, None) == ctr.CTR_EINVAL


def test_struct_layout_matches_header(tmp_path):
    from paper_2609_16206_gb300 import ctr
    structs = {"ctr_requests": ctr.CtrRequests, "ctr_trace_cfg": ctr.CtrTraceCfg, "ctr_sim_cfg": ctr.CtrSimCfg,
               "ctr_cost_consts": ctr.CtrCostConsts}
    lines = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"', "int main(void){"]
    for cname, py in structs.items():
        lines.append(f'printf("{cname} sizeof %zu\\n", sizeof({cname}));')
        for field, _ in py._fields_:
            lines.append(f'printf("{cname} {field} %zu\\n", offsetof({cname}, {field}));')
    lines.append("return 0;}")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-o", str(exe), str(src)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {tuple(l.split()[:2]): int(l.split()[2]) for l in out if l.strip()}
    for cname, py in structs.items():
        assert got[(cname, "sizeof")] == ctypes.sizeof(py), cname
        for field, _ in py._fields_:
            assert got[(cname, field)] == getattr(py, field).offset, (cname, field)


def test_product_path_fails_loudly_without_cuda():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2609_16206_gb300 import ctr
    from paper_2609_16206_gb300 import workloads as W
    with pytest.raises(Exception):
        tr = ctr.empty_requests(1, 10, "cpu")
        ctr.ctr_gen_trace(W.TraceCfg(), 1, 0, 10, tr)


def test_workspace_query_without_gpu_is_zero():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2609_16206_gb300 import ctr
    from paper_2609_16206_gb300 import workloads as W
    assert ctr.ctr_workspace_bytes(0, W.SimCfg(), 4, 100) == 0


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """Without a built libctr.so the first call raises at once (it must not
    fall back, and must not block on the loader's own lock)."""
    import threading

    from paper_2609_16206_gb300 import ctr
    monkeypatch.setattr(ctr, "LIB_PATH", str(tmp_path / "libctr.so"))
    monkeypatch.setattr(ctr, "_lib", None)
    out = {}

    def call():
        try:
            ctr.lib()
        except ctr.CtrError as e:
            out["err"] = e

    t = threading.Thread(target=call, daemon=True)
    t.start()
    t.join(timeout=20)
    assert not t.is_alive(), "loading a missing library blocked"
    assert "err" in out and "is missing" in str(out["err"])
    assert ctr.ctr_strerror(ctr.CTR_EINVAL) == "libctr.so not loaded"


def test_binding_switches_between_the_two_libraries():
    """ctr.use_library loads the bounds-checked twin and back (no device calls)."""
    from paper_2609_16206_gb300 import build, ctr
    build.build()
    checked = build.build(checked=True)
    before = ctr.use_library(checked)
    try:
        assert ctr.ctr_bounds_checked() == 1 and ctr.ctr_abi_version() == 8
    finally:
        ctr.use_library(before)
    assert ctr.LIB_PATH == before and ctr.ctr_bounds_checked() == 0
