"""ctr_simulate_noalloc, the allocation-free variant of ctr_simulate.

It exists for callers that cannot allocate device memory (a plugin inside a
serving process whose pool owns the GPU, code between another component's
stream-capture calls, a loop that must never reach the driver's allocator):
its scratch is a fixed array inside the library.  This file is collected
last on purpose, and the test passes both on its own in a fresh process and
after every other test.  It calls the entry point through the C ABI twice in
a row -- the second call reuses the array the first one left behind -- and
requires both to match ctr_simulate with a caller-provided workspace exactly
(every routing decision, time, row hash and status, the simulator's
bit-exact tolerance)."""
import numpy as np
import pytest
import torch

from gpuutil import gen, need_gpu, simulate
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _noalloc(ctr, sc, sets, pols, tr, R, N):
    rows = R * len(sets) * len(pols)
    out = {"t_first_us": torch.full((rows, N), -7, dtype=torch.int64, device="cuda"),
           "t_done_us": torch.full((rows, N), -7, dtype=torch.int64, device="cuda"),
           "hash": torch.zeros(rows, dtype=torch.int64, device="cuda"),
           "status": torch.full((rows,), 99, dtype=torch.int32, device="cuda"),
           "i_pre": torch.full((rows, N), 255, dtype=torch.uint8, device="cuda"),
           "i_dec": torch.full((rows, N), 255, dtype=torch.uint8, device="cuda")}
    ctr.ctr_simulate_noalloc(sc, sets, pols, tr, R, N, out["t_first_us"], out["t_done_us"], out["hash"],
                             out["status"], i_pre=out["i_pre"], i_dec=out["i_dec"])
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["hash"] = res["hash"].astype(np.uint64)
    return res


@pytest.mark.parametrize("wl,R,N", [(W.replica_sweep(), 40, 2500), (W.large_pool(rate_mreq=34_000), 2, 2000)])
def test_noalloc_matches_workspace_entry_twice(wl, R, N):
    ctr = need_gpu()
    tr = gen(ctr, wl.trace, R, N)
    sets, pols = [wl.consts[0]], list(W.ALL_POLICIES)
    ref = simulate(ctr, wl.sim, sets, pols, tr, R, N)
    assert (ref["status"] == 0).all()
    for call in range(2):
        got = _noalloc(ctr, wl.sim, sets, pols, tr, R, N)
        for key in ("t_first_us", "t_done_us", "i_pre", "i_dec", "hash", "status"):
            assert np.array_equal(got[key], ref[key]), (call, key)


def test_noalloc_rejects_structures_beyond_its_array():
    ctr = need_gpu()
    sc = W.replica_sweep().sim.replace(cap_pending=1 << 20, cap_waiting=1 << 20, cap_active=1 << 20)
    tr = gen(ctr, W.replica_sweep().trace, 1, 10)
    with pytest.raises(ctr.CtrError) as err:
        _noalloc(ctr, sc, [W.CALIBRATED], [0], tr, 1, 10)
    assert err.value.code == ctr.CTR_EINVAL
