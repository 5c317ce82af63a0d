"""Parity: the GPU trace generator is bit-identical to the CPU oracle."""
import numpy as np
import pytest

from gpuutil import gen, need_gpu
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _compare(orc, tc, tr, n_replicas, n_req, offset=0, rows=None):
    rows = range(n_replicas) if rows is None else rows
    for r in rows:
        ref = orc.gen_trace(tc, n_req, replica=offset + r)
        for key, val in ref.items():
            got = tr[key][r].cpu().numpy()
            assert np.array_equal(got, val), (key, r, np.flatnonzero(got != val)[:5])


@pytest.mark.parametrize("name,tc,R,N,off", [
    ("single_replica", W.single_replica().trace, 1, 2000, 0),
    ("bursty_mmpp_3seeds", W.replica_sweep().trace, 24, 3000, 0),
    ("bursty_offset", W.replica_sweep().trace, 5, 1000, 4091),
    ("three_classes_noise06", W.large_pool(rate_mreq=30_000).trace, 6, 5000, 0),
    ("ragged_33", W.TraceCfg(seed=99), 3, 33, 0),
    ("ragged_1", W.TraceCfg(seed=5), 2, 1, 0),
    ("ragged_1007", W.TraceCfg(seed=6, noise_sigma=0.0, n_classes=1, class_thr=()), 2, 1007, 7),
    ("homogeneous_chat", W.TraceCfg(mix_short_thr=W.prob_to_u32_threshold(1.0)), 2, 700, 0),
    ("all_reasoning", W.TraceCfg(mix_short_thr=0, seed=2**40 + 17), 2, 700, 0),
])
def test_trace_bit_identical(orc, name, tc, R, N, off):
    ctr = need_gpu()
    tr = gen(ctr, tc, R, N, off)
    _compare(orc, tc, tr, R, N, off)


def test_empty_sizes(orc):
    ctr = need_gpu()
    gen(ctr, W.TraceCfg(), 0, 100)
    gen(ctr, W.TraceCfg(), 3, 0)


def test_invalid_trace_cfg_rejected():
    ctr = need_gpu()
    tr = ctr.empty_requests(1, 10, "cuda")
    for bad in (W.TraceCfg(n_seeds=0), W.TraceCfg(rate_mreq=(0, 0)), W.TraceCfg(arrival_kind=2),
                W.TraceCfg(prompt_min=100, prompt_max=50), W.TraceCfg(noise_sigma=-1.0),
                W.TraceCfg(n_classes=5), W.TraceCfg(prompt_mu=float("nan"))):
        with pytest.raises(ctr.CtrError):
            ctr.ctr_gen_trace(bad, 1, 0, 10, tr)


def test_full_size_sweep_sampled(orc):
    """The benchmarked replica sweep, 4,096 replicas x 20,000 requests, generated
    in one launch; sampled replicas (each seed, first and last) against the oracle."""
    ctr = need_gpu()
    wl = W.replica_sweep()
    tr = gen(ctr, wl.trace, wl.n_replicas, wl.n_req)
    _compare(orc, wl.trace, tr, wl.n_replicas, wl.n_req, rows=[0, 1, 2, 1366, 2731, 4095])
