"""Compile libctr.so (the CUDA library behind include/ctr.h) in-tree for sm_103a.

Each translation unit compiles in parallel with nvcc; the trace unit is built
with -fmad=false so that no fp32 product is fused into an add (the trace is
defined in fp32, each operation rounded on its own, and must be bit-identical
to the CPU construction, which is compiled with -ffp-contract=off).  Outputs: csrc/../_build/*.o and
libctr.so next to this file (both git-ignored).

build(checked=True) compiles the same sources with CTR_BOUNDS_CHECK=1 into
_build_checked/ and libctr_checked.so: the simulator then checks every index
into its workspace, the trace and the outputs (see ctr_bounds_checked in
include/ctr.h).  build_all() makes both libraries from one pool of jobs.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OBJ = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libctr.so")
OBJ_CHECKED = os.path.join(HERE, "_build_checked")
LIB_CHECKED = os.path.join(HERE, "libctr_checked.so")
SOURCES = ["api.cu", "trace.cu", "sim.cu", "score.cu", "goodput.cu", "noalloc.cu"]
HEADERS = [os.path.join(CSRC, "ctr_internal.cuh"), os.path.join(ROOT, "include", "ctr.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
          "-I", os.path.join(ROOT, "include")]
PER_FILE = {"trace.cu": ["-fmad=false"]}


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found; the CUDA toolkit is required to build libctr.so")
    return path


def _stale(target: str, deps) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _jobs(checked: bool, force: bool, ptxas_info: bool):
    """(compile commands still to run, object files, library path) of one library."""
    obj_dir, lib = (OBJ_CHECKED, LIB_CHECKED) if checked else (OBJ, LIB)
    os.makedirs(obj_dir, exist_ok=True)
    cc = nvcc()
    objs, jobs = [], []
    for src in SOURCES:
        s = os.path.join(CSRC, src)
        o = os.path.join(obj_dir, src.replace(".cu", ".o"))
        objs.append(o)
        if force or _stale(o, [s] + HEADERS):
            cmd = [cc] + ARCH + COMMON + PER_FILE.get(src, []) + (["-DCTR_BOUNDS_CHECK=1"] if checked else []) + \
                  (["-Xptxas", "-v"] if ptxas_info else []) + ["-c", s, "-o", o]
            jobs.append(cmd)
    return jobs, objs, lib


def _run(jobs, verbose: bool, ptxas_info: bool):
    if not jobs:
        return
    with cf.ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 4)) as ex:
        results = list(ex.map(lambda c: subprocess.run(c, capture_output=True, text=True), jobs))
    for cmd, r in zip(jobs, results):
        if verbose or ptxas_info or r.returncode != 0:
            sys.stderr.write(r.stdout + r.stderr)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed: " + " ".join(cmd))


def _link(objs, lib, relink: bool):
    if relink or _stale(lib, objs):
        tmp = lib + f".tmp{os.getpid()}"
        r = subprocess.run([nvcc()] + ARCH + ["-shared", "-o", tmp] + objs, capture_output=True, text=True)
        if r.returncode != 0:
            sys.stderr.write(r.stdout + r.stderr)
            raise RuntimeError("nvcc link failed")
        os.replace(tmp, lib)


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False, checked: bool = False) -> str:
    jobs, objs, lib = _jobs(checked, force, ptxas_info)
    _run(jobs, verbose, ptxas_info)
    _link(objs, lib, force or bool(jobs))
    return lib


def build_all(force: bool = False, verbose: bool = False) -> tuple:
    """libctr.so and libctr_checked.so, their translation units compiled in one pool."""
    plain = _jobs(False, force, False)
    checked = _jobs(True, force, False)
    _run(plain[0] + checked[0], verbose, False)
    _link(plain[1], plain[2], force or bool(plain[0]))
    _link(checked[1], checked[2], force or bool(checked[0]))
    return plain[2], checked[2]


if __name__ == "__main__":
    if "--all" in sys.argv:
        print(*build_all(force="--force" in sys.argv, verbose=True))
    else:
        print(build(force="--force" in sys.argv, verbose=True, ptxas_info="--ptxas" in sys.argv,
                    checked="--checked" in sys.argv))
