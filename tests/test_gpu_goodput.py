"""Parity: GPU goodput (SLO-met count, nearest-rank P99 TTFT) equals the oracle's."""
import numpy as np
import pytest
import torch

from gpuutil import gen, host_trace, need_gpu, simulate, to_dev
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _goodput(ctr, sc, tr, R, rows_per, N, tf, td):
    rows = R * rows_per
    met = torch.full((rows,), -5, dtype=torch.int64, device="cuda")
    p99 = torch.full((rows,), -5, dtype=torch.int64, device="cuda")
    ctr.ctr_goodput(sc, tr, R, rows_per, N, tf, td, met, p99)
    torch.cuda.synchronize()
    return met.cpu().numpy(), p99.cpu().numpy()


@pytest.mark.parametrize("wl,R,N", [(W.single_replica(), 1, 2000), (W.replica_sweep(), 8, 5000),
                                    (W.large_pool(rate_mreq=34_000), 2, 3000), (W.replica_sweep(), 3, 37),
                                    (W.replica_sweep(), 1, 45_000)])  # rows past the shared-memory staging
def test_goodput_matches_oracle(orc, wl, R, N):
    ctr = need_gpu()
    tr = gen(ctr, wl.trace, R, N)
    pols = list(W.ALL_POLICIES)
    res = simulate(ctr, wl.sim, [wl.consts[0]], pols, tr, R, N)
    tf = torch.from_numpy(res["t_first_us"]).cuda()
    td = torch.from_numpy(res["t_done_us"]).cuda()
    met, p99 = _goodput(ctr, wl.sim, tr, R, len(pols), N, tf, td)
    for r in range(R):
        trh = host_trace(tr, r)
        for j in range(len(pols)):
            row = r * len(pols) + j
            assert (met[row], p99[row]) == orc.goodput(wl.sim, trh, res["t_first_us"][row], res["t_done_us"][row])


def test_goodput_adversarial_times(orc):
    """Equal values, huge spreads and negative TTFTs exercise every radix digit."""
    ctr = need_gpu()
    rng = np.random.default_rng(8)
    sc = W.SimCfg(n_classes=3, ttft_slo_us=(10, 10**6, 10**12), tpot_slo_us=(0, 5, 10**9))
    for N in (1, 2, 100, 101, 4097, 45_000):  # 45,000: rows too long to stage in shared memory
        R = 3
        trh = {"arrival_us": np.sort(rng.integers(0, 10**6, (R, N)), axis=1), "prompt_len": np.ones((R, N)),
               "true_out": rng.integers(1, 4, (R, N)), "pred_out": np.ones((R, N)),
               "slo_class": rng.integers(0, 5, (R, N))}
        tf = trh["arrival_us"] + rng.choice([0, 7, 10**6, 2**45, -3], size=(R, N))
        tf[1] = trh["arrival_us"][1] + 42                     # all equal TTFT
        td = tf + rng.integers(0, 20, (R, N))
        tr = to_dev(trh)
        met, p99 = _goodput(ctr, sc, tr, R, 1, N, torch.from_numpy(tf).cuda(), torch.from_numpy(td).cuda())
        for r in range(R):
            row = {k: v[r] for k, v in trh.items()}
            assert (met[r], p99[r]) == orc.goodput(sc, row, tf[r], td[r]), (N, r)


def test_goodput_empty(orc):
    ctr = need_gpu()
    tr = ctr.empty_requests(2, 0, "cuda")
    z = torch.empty((2, 0), dtype=torch.int64, device="cuda")
    met, p99 = _goodput(ctr, W.SimCfg(), tr, 2, 1, 0, z, z)
    assert met.tolist() == [0, 0] and p99.tolist() == [-1, -1]
