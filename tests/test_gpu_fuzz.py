"""Parity across the configuration space: seeded random cluster shapes,
capacities, physics, cost constants (with ablation, ledger backlog and polled
occupancy), policies, batched prefill and trace laws, each simulated on the
GPU and by the oracle, compared row by row (status, checksum, and every time
and route)."""
import numpy as np
import pytest
import torch

from gpuutil import gen, host_trace, need_gpu, simulate
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _case(rng):
    n_pre = int(rng.integers(1, 5))
    n_dec = int(rng.integers(1, 13))
    n_classes = int(rng.integers(1, 5))
    kv_cap = int(rng.choice([9_000, 20_000, 60_000, 200_000]))
    sc = W.SimCfg(
        n_prefill=n_pre, n_decode=n_dec, kv_cap_tokens=kv_cap,
        pre_base_us=int(rng.integers(1, 40_000)), pre_us_per_tok=int(rng.integers(0, 300)),
        xfer_us_per_tok=int(rng.integers(0, 50)), dec_base_us=int(rng.integers(1, 30_000)),
        dec_us_per_seq=int(rng.integers(0, 500)), dec_kv_tokens_per_us=int(rng.choice([1, 7, 1000, 1 << 20])),
        n_classes=n_classes, ttft_slo_us=tuple(int(x) for x in rng.integers(10_000, 5_000_000, 4)),
        tpot_slo_us=tuple(int(x) for x in rng.integers(1_000, 300_000, 4)),
        cap_pending=int(rng.choice([8, 1024, 1024])), cap_waiting=int(rng.choice([8, 1024, 1024])),
        cap_active=int(rng.choice([16, 1024, 1024])), cap_prefill_ring=int(rng.choice([16, 1024, 1024])),
        heuristic_threshold_tokens=int(rng.integers(0, 2048)),
        prefill_batch_tokens=int(rng.choice([0, 0, 1, 2048, 8192])))
    mix = float(rng.random())
    tc = W.TraceCfg(seed=int(rng.integers(0, 1 << 40)), arrival_kind=int(rng.integers(0, 2)),
                    rate_mreq=(int(rng.integers(500, 15_000)), int(rng.integers(500, 25_000))),
                    dwell_mean_us=int(rng.integers(100_000, 20_000_000)), prompt_max=min(4096, kv_cap // 2),
                    mix_short_thr=W.prob_to_u32_threshold(mix), noise_sigma=float(rng.choice([0.0, 0.3, 1.2])),
                    n_classes=n_classes,
                    class_thr=tuple(sorted(W.prob_to_u32_threshold(float(x)) for x in rng.random(n_classes - 1))))
    sets = []
    for _ in range(int(rng.integers(1, 4))):
        sets.append(W.CostConsts(
            tau_pre0_us=int(rng.integers(0, 50_000)), tau_pre_us=int(rng.integers(0, 400)),
            tau_dec_us=int(rng.integers(0, 40_000)), w_q_us=int(rng.integers(0, 20_000)),
            w_b_q8=int(rng.integers(0, 1024)), w_s_q8=int(rng.integers(0, 1024)), rho_q8=int(rng.integers(0, 1024)),
            sigma_q8=tuple(int(x) for x in rng.integers(0, 1024, 4)), ablate=int(rng.integers(0, 8)),
            proxy_backlog=int(rng.integers(0, 2)), poll_us=int(rng.choice([0, 0, 1_000, 50_000, 1 << 30]))))
    pols = [int(p) for p in rng.permutation(5)[:int(rng.integers(1, 6))]]
    n_req = int(rng.choice([1, 31, 257, 1200]))
    n_rep = int(rng.integers(1, 4))
    return sc, tc, sets, pols, n_rep, n_req


@pytest.mark.parametrize("seed", range(160))
def test_random_configuration(orc, seed):
    ctr = need_gpu()
    rng = np.random.default_rng(10_000 + seed)
    sc, tc, sets, pols, R, N = _case(rng)
    tr = gen(ctr, tc, R, N)
    res = simulate(ctr, sc, sets, pols, tr, R, N)
    rows = R * len(sets) * len(pols)
    met = torch.empty(rows, dtype=torch.int64, device="cuda")
    p99 = torch.empty(rows, dtype=torch.int64, device="cuda")
    ctr.ctr_goodput(sc, tr, R, len(sets) * len(pols), N, torch.from_numpy(res["t_first_us"]).cuda(),
                    torch.from_numpy(res["t_done_us"]).cuda(), met, p99)
    met, p99 = met.cpu().numpy(), p99.cpu().numpy()
    row = 0
    for r in range(R):
        trh = host_trace(tr, r)
        ref_tr = orc.gen_trace(tc, N, replica=r)
        for key in ref_tr:
            assert np.array_equal(trh[key], ref_tr[key]), (seed, key)
        for cc in sets:
            for pol in pols:
                o = orc.simulate(sc, cc, pol, trh)
                assert res["status"][row] == o["status"], (seed, row, res["status"][row], o["status"])
                if o["status"] == 0:
                    assert int(res["hash"][row]) == o["hash"], (seed, row)
                    for key in ("t_first_us", "t_done_us", "i_pre", "i_dec"):
                        assert np.array_equal(res[key][row], o[key]), (seed, row, key)
                    assert (met[row], p99[row]) == orc.goodput(sc, trh, o["t_first_us"], o["t_done_us"]), (seed, row)
                row += 1
