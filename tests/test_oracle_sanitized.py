"""The oracle built with AddressSanitizer and UndefinedBehaviorSanitizer.

A separate build of oracle/ctr_oracle.c with -fsanitize=address,undefined
(every report fatal) runs in a child process: the hand-derived worked traces
under every policy, a 2,000-request replica-sweep row under every policy
(with the proxy's signals and the ablation mask on one set), a batched-prefill
row, the goodput scorer on each, the fp64 scorer on a small batch, and the
input and capacity errors.  The child must exit cleanly and its results must
equal the plain build's, computed here."""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

import simutil as U
from conftest import ROOT
from paper_2609_16206_gb300 import workloads as W

CHILD = r'''
import json, sys
import numpy as np
sys.path.insert(0, sys.argv[2]); sys.path.insert(0, sys.argv[3])
import oracle
oracle._LIB_PATH = sys.argv[1]   # the sanitized build, already compiled
import simutil as U
from paper_2609_16206_gb300 import workloads as W
from test_oracle_sanitized import cases
out = []
for sc, cc, pol, tr in cases(oracle):
    r = oracle.simulate(sc, cc, pol, tr)
    g = oracle.goodput(sc, tr, r["t_first_us"], r["t_done_us"]) if r["status"] == 0 else None
    out.append([r["status"], r["hash"], g])
p, oh, cls = W.score_requests(257, seed=3)
Q, A, kap = W.score_state(19, seed=4)
am, best, second = oracle.score_batch(p, oh, cls, Q, A, kap, W.SCORE_CONSTS)
out.append([am.tolist(), best.tolist()])
print(json.dumps(out))
'''


def cases(orc):
    """(sim cfg, constants, policy, trace) of every run, in a fixed order."""
    runs = []
    for case in U.worked_traces():
        sc, cc, tr = U.sim_from(case["sim"]), U.consts_from(case["consts"]), U.trace_from(case["requests"])
        runs += [(sc, cc, pol, tr) for pol in W.ALL_POLICIES + (W.POLICY_LEARNED_P2,)]
    wl = W.replica_sweep()
    tr = orc.gen_trace(wl.trace, 2000, replica=5)
    for cc in (W.CALIBRATED, W.as_deployed(W.CALIBRATED).replace(ablate=W.ABLATE_SLO)):
        runs += [(wl.sim, cc, pol, tr) for pol in W.ALL_POLICIES + (W.POLICY_LEARNED_P2,)]
    doc = W.document(n_replicas=1, n_req=1500)
    dtr = orc.gen_trace(doc.trace, 1500, replica=0)
    runs += [(doc.sim, W.CALIBRATED, pol, dtr) for pol in W.ALL_POLICIES]
    # the error paths: a tiny waiting FIFO, a small step budget, a request that breaks the bounds
    runs.append((wl.sim.replace(cap_waiting=2, cap_pending=2), W.CALIBRATED, W.POLICY_RR, tr))
    runs.append((wl.sim.replace(max_steps_per_instance=500), W.CALIBRATED, W.POLICY_LEARNED, tr))
    bad = {k: v.copy() for k, v in tr.items()}
    bad["true_out"][7] = 0
    runs.append((wl.sim, W.CALIBRATED, W.POLICY_JSQ, bad))
    return runs


def _sanitizer_flags():
    return ["-fsanitize=address,undefined", "-fno-sanitize-recover=all", "-fno-omit-frame-pointer", "-g", "-O1"]


def test_oracle_under_address_and_undefined_sanitizers(orc, tmp_path):
    so = str(tmp_path / "liboracle_san.so")
    src = os.path.join(ROOT, "oracle", "ctr_oracle.c")
    r = subprocess.run(["gcc", "-std=gnu11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-Wall"]
                       + _sanitizer_flags() + ["-o", so, src, "-lm"], capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("gcc cannot build with -fsanitize=address,undefined here: " + r.stderr[-300:])
    asan = subprocess.run(["gcc", "-print-file-name=libasan.so"], capture_output=True, text=True).stdout.strip()
    if not os.path.isabs(asan) or not os.path.exists(asan):
        pytest.skip("libasan.so not found")
    env = dict(os.environ, LD_PRELOAD=asan, ASAN_OPTIONS="detect_leaks=0:abort_on_error=1",
               UBSAN_OPTIONS="print_stacktrace=1:halt_on_error=1")
    child = subprocess.run([sys.executable, "-c", CHILD, so, ROOT, os.path.join(ROOT, "tests")],
                           capture_output=True, text=True, env=env, timeout=600)
    assert child.returncode == 0, child.stderr[-3000:]
    assert "runtime error" not in child.stderr and "AddressSanitizer" not in child.stderr, child.stderr[-3000:]
    got = json.loads(child.stdout.strip().splitlines()[-1])

    want = []
    for sc, cc, pol, tr in cases(orc):
        res = orc.simulate(sc, cc, pol, tr)
        g = list(orc.goodput(sc, tr, res["t_first_us"], res["t_done_us"])) if res["status"] == 0 else None
        want.append([res["status"], res["hash"], g])
    p, oh, cls = W.score_requests(257, seed=3)
    Q, A, kap = W.score_state(19, seed=4)
    am, best, _ = orc.score_batch(p, oh, cls, Q, A, kap, W.SCORE_CONSTS)
    assert got[:-1] == want
    assert got[-1][0] == am.tolist() and np.array_equal(np.array(got[-1][1]), best)
    statuses = {w[0] for w in want}
    assert {0, orc.EINVAL, orc.EOVERFLOW, orc.ETIMEOUT} <= statuses   # every error path ran
