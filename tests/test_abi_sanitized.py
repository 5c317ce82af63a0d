"""The C ABI's host-side argument validation under AddressSanitizer and
UndefinedBehaviorSanitizer (no GPU needed).

A separate build of libctr.so whose host code is instrumented with
-fsanitize=address,undefined (every report fatal) is loaded in a child
process, which calls every entry point with each configuration field at,
just past and far past its bounds (64-bit extremes, NaN and infinite
parameters, null pointers, zero and negative sizes) and with a few thousand
seeded random configurations.  Each call must return one of the documented
codes -- CTR_EINVAL where an argument is out of range, and without a GPU
CTR_ECUDA (or 0 for an empty launch) where every argument is valid -- and the
child must exit cleanly."""
import os
import subprocess
import sys

import pytest

from conftest import ROOT

CHILD = r'''
import ctypes as C, math, sys
import numpy as np
sys.path.insert(0, sys.argv[2])
from paper_2609_16206_gb300 import ctr
from paper_2609_16206_gb300 import workloads as W
ctr.LIB_PATH = sys.argv[1]
L = ctr.lib()
OK, EINVAL, ECUDA = ctr.CTR_OK, ctr.CTR_EINVAL, ctr.CTR_ECUDA
I64 = [-(1 << 63), -(1 << 40), -1, 0, 1, (1 << 20) + 1, (1 << 31), (1 << 39), (1 << 40) + 1, (1 << 63) - 1]
I32 = [-(1 << 31), -1, 0, 1, 33, (1 << 20) + 1, (1 << 31) - 1]
F64 = [float("nan"), float("inf"), -float("inf"), -1.0, 0.0, 1e300]
dummy = (C.c_uint8 * 64)()
ptr = C.cast(dummy, C.c_void_p)
req = ctr.CtrRequests(ptr, ptr, ptr, ptr, ptr)
seen = set()

def rc(v):
    assert v in (OK, EINVAL, ECUDA), v
    seen.add(v)
    return v

def sim_call(cfg, cc=None, n_sets=1, pols=(0,), n_rep=1, n_req=10, ws_bytes=1 << 20, noalloc=False):
    sets = ctr.consts_array([cc or W.CALIBRATED] * max(n_sets, 1)) if cc is None or not isinstance(cc, C.Array) else cc
    pa = (C.c_int32 * max(len(pols), 1))(*pols)
    if noalloc:
        return rc(L.ctr_simulate_noalloc(C.byref(cfg), sets, n_sets, pa, len(pols), req, n_rep, n_req, ptr, ptr, ptr,
                                         ptr, ptr, ptr, None))
    goodput = (ptr, ptr) if n_rep % 2 else (None, None)
    return rc(L.ctr_simulate(C.byref(cfg), sets, n_sets, pa, len(pols), req, n_rep, n_req, ptr, ptr, ptr, ptr, ptr,
                             ptr, *goodput, ptr, ws_bytes, None))

# every simulator field at its extremes, one at a time
base = ctr.sim_cfg_struct(W.replica_sweep().sim)
for name, typ in ctr.CtrSimCfg._fields_:
    vals = I64 if typ in (C.c_int64,) else I32
    if hasattr(typ, "_length_"):
        continue
    for v in vals:
        cfg = ctr.sim_cfg_struct(W.replica_sweep().sim)
        setattr(cfg, name, v)
        sim_call(cfg)
        sim_call(cfg, noalloc=True)
        rc(0 if L.ctr_workspace_bytes(0, C.byref(cfg), 4, 10) == 0 else OK)
# constant sets
for name, typ in ctr.CtrCostConsts._fields_:
    if hasattr(typ, "_length_"):
        continue
    for v in (I64 if typ == C.c_int64 else I32):
        cs = ctr.consts_array([W.CALIBRATED])
        try:
            setattr(cs[0], name, v)
        except (OverflowError, TypeError):
            continue
        sim_call(base, cc=cs)
for n_sets in (-1, 0, 1, 129):
    sim_call(base, cc=ctr.consts_array([W.CALIBRATED] * 130), n_sets=n_sets)
for pols in ((), (0, 1, 2, 3, 4, 0), (-1,), (5,), (4, 3)):
    if pols:
        sim_call(base, pols=pols)
for n_rep, n_req in ((-1, 10), (0, 10), (1, -1), (1, (1 << 23) + 1), ((1 << 31) - 1, 1 << 23), (1, 0)):
    sim_call(base, n_rep=n_rep, n_req=n_req)
for wsb in (0, 255, 256, 1 << 40):
    sim_call(base, ws_bytes=wsb)
# trace generator
def trace_call(cfg, n_rep=2, off=0, n_req=10, out=req):
    return rc(L.ctr_gen_trace(C.byref(cfg), n_rep, off, n_req, out, None))
for name, typ in ctr.CtrTraceCfg._fields_:
    if hasattr(typ, "_length_"):
        continue
    vals = F64 if typ == C.c_double else (I64 if typ in (C.c_int64, C.c_uint64) else I32)
    for v in vals:
        cfg = ctr.trace_cfg_struct(W.replica_sweep().trace)
        try:
            setattr(cfg, name, v if typ != C.c_uint64 else v % (1 << 64))
        except (OverflowError, TypeError):
            continue
        trace_call(cfg)
tc = ctr.trace_cfg_struct(W.replica_sweep().trace)
for n_rep, off, n_req in ((-1, 0, 1), (1, -1, 1), (1, (1 << 63) - 1, 1), ((1 << 31) - 1, (1 << 40), 1), (1, 0, -1),
                          (1, 0, (1 << 23) + 1), (0, 0, 5), (3, 0, 0)):
    trace_call(tc, n_rep, off, n_req)
trace_call(tc, out=ctr.CtrRequests())
# scorer
cv = (C.c_float * 13)(*W.SCORE_CONSTS)
for n_req, n_inst in ((-1, 4), (0, 4), (10, 0), (10, 257), (10, -5), (1 << 40, 64)):
    rc(L.ctr_score_batch(ptr, ptr, ptr, n_req, ptr, ptr, ptr, n_inst, cv, ptr, ptr, None, None))
for i in range(13):
    for v in (float("nan"), float("inf"), -1.0):
        bad = (C.c_float * 13)(*W.SCORE_CONSTS)
        bad[i] = v
        rc(L.ctr_score_batch(ptr, ptr, ptr, 10, ptr, ptr, ptr, 4, bad, ptr, ptr, None, None))
rc(L.ctr_score_batch(None, ptr, ptr, 10, ptr, ptr, ptr, 4, cv, ptr, ptr, None, None))
rc(L.ctr_score_batch(ptr, ptr, ptr, 10, ptr, ptr, ptr, 4, None, ptr, ptr, None, None))
# goodput
for n_rep, rows_per, n_req in ((-1, 4, 10), (1, 0, 10), (1, 4, -1), ((1 << 31) - 1, (1 << 31) - 1, 1), (0, 4, 10)):
    rc(L.ctr_goodput(C.byref(base), req, n_rep, rows_per, n_req, ptr, ptr, ptr, ptr, None, None))
rc(L.ctr_goodput(None, req, 1, 4, 10, ptr, ptr, ptr, ptr, None, None))
# seeded random configurations
rng = np.random.default_rng(1)
pick = lambda xs: xs[int(rng.integers(len(xs)))]
for _ in range(3000):
    cfg = ctr.sim_cfg_struct(W.replica_sweep().sim)
    for name, typ in ctr.CtrSimCfg._fields_:
        if not hasattr(typ, "_length_") and rng.random() < 0.3:
            setattr(cfg, name, pick(I64 if typ == C.c_int64 else I32))
    cs = ctr.consts_array([W.CALIBRATED])
    for name, typ in ctr.CtrCostConsts._fields_:
        if not hasattr(typ, "_length_") and rng.random() < 0.2:
            try:
                setattr(cs[0], name, pick(I64 if typ == C.c_int64 else I32))
            except (OverflowError, TypeError):
                pass
    sim_call(cfg, cc=cs, n_rep=pick([0, 1, 3]), n_req=pick([0, 7, 1 << 23]))
    tcfg = ctr.trace_cfg_struct(W.replica_sweep().trace)
    for name, typ in ctr.CtrTraceCfg._fields_:
        if not hasattr(typ, "_length_") and rng.random() < 0.2:
            v = pick(F64) if typ == C.c_double else pick(I64 if typ in (C.c_int64, C.c_uint64) else I32)
            try:
                setattr(tcfg, name, v if typ != C.c_uint64 else v % (1 << 64))
            except (OverflowError, TypeError):
                pass
    trace_call(tcfg, pick([0, 1, 2]), pick([0, 5, (1 << 40) - 3]), pick([0, 3]))
assert L.ctr_abi_version() == 8
for code in range(-6, 3):
    assert L.ctr_strerror(code)
print("seen", sorted(seen))
'''


def test_c_abi_validation_under_sanitizers(tmp_path):
    import shutil
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    csrc = os.path.join(ROOT, "paper_2609_16206_gb300", "csrc")
    # one flag per -Xcompiler: nvcc splits its arguments at commas
    san = ["-Xcompiler", "-fsanitize=address", "-Xcompiler", "-fsanitize=undefined",
           "-Xcompiler", "-fno-sanitize-recover=all", "-Xcompiler", "-fno-omit-frame-pointer"]
    common = ["-gencode", "arch=compute_103a,code=sm_103a", "-O1", "-std=c++17", "-Xcompiler", "-fPIC",
              "-I", os.path.join(ROOT, "include")] + san
    objs, procs = [], []
    for src in ("api.cu", "trace.cu", "sim.cu", "score.cu", "goodput.cu", "noalloc.cu"):
        o = str(tmp_path / src.replace(".cu", ".o"))
        objs.append(o)
        procs.append(subprocess.Popen([nvcc] + common + ["-c", os.path.join(csrc, src), "-o", o],
                                      stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True))
    for p in procs:
        out, _ = p.communicate()
        if p.returncode != 0:
            pytest.skip("sanitized build failed: " + out[-400:])
    so = str(tmp_path / "libctr_san.so")
    r = subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-shared", "-o", so] + objs + san,
                       capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("sanitized link failed: " + r.stderr[-400:])
    asan = subprocess.run(["gcc", "-print-file-name=libasan.so"], capture_output=True, text=True).stdout.strip()
    if not os.path.isabs(asan) or not os.path.exists(asan):
        pytest.skip("libasan.so not found")
    env = dict(os.environ, LD_PRELOAD=asan, CUDA_VISIBLE_DEVICES="",
               ASAN_OPTIONS="detect_leaks=0:abort_on_error=1:protect_shadow_gap=0",
               UBSAN_OPTIONS="print_stacktrace=1:halt_on_error=1")
    child = subprocess.run([sys.executable, "-c", CHILD, so, ROOT], capture_output=True, text=True, env=env,
                           timeout=900)
    assert child.returncode == 0, child.stdout[-2000:] + child.stderr[-4000:]
    assert "runtime error" not in child.stderr and "AddressSanitizer" not in child.stderr, child.stderr[-4000:]
    assert "seen [-2, -1, 0]" in child.stdout, child.stdout
