"""Parity: GPU goodput (SLO-met count, nearest-rank P99 TTFT and P99 TPOT) equals the oracle's."""
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


@pytest.mark.parametrize("crowd", [1, 511, 512, 513, 3000])
def test_goodput_crowded_p99_bin(orc, crowd):
    """The P99's rank falls among `crowd` requests whose TTFTs share one
    logarithmic bin: up to 512 of them are counted out exactly in shared
    memory, more go to the radix select; TTFTs at 0 and 2^32 - 1 (the ends of
    the binned range) and a row with one TTFT of 2^32 (outside it) ride along."""
    ctr = need_gpu()
    rng = np.random.default_rng(crowd)
    R, below = 3, 3500
    above = max(1, (crowd + below) // 99 - crowd // 3)
    N = below + crowd + above
    rank = (99 * N + 99) // 100 - 1
    ttft = np.concatenate([rng.integers(0, 1000, below), 10**6 + rng.integers(0, 2000, crowd),
                           rng.integers(10**9, 2**32, above)])
    ttft[0], ttft[-1] = 0, 2**32 - 1
    srt = np.sort(ttft)
    if crowd > 1:
        assert 10**6 <= srt[rank] < 10**6 + 2000, "the P99 must lie in the crowded bin"
    tf = np.empty((R, N), dtype=np.int64)
    arr = np.sort(rng.integers(0, 10**7, (R, N)), axis=1)
    for r in range(R):
        tf[r] = arr[r] + rng.permutation(ttft)
    tf[2, N // 2] = arr[2, N // 2] + 2**32  # outside [0, 2^32): the whole row takes the radix select
    trh = {"arrival_us": arr, "prompt_len": np.ones((R, N)), "true_out": rng.integers(1, 4, (R, N)),
           "pred_out": np.ones((R, N)), "slo_class": rng.integers(0, 4, (R, N))}
    td = tf + rng.integers(0, 20, (R, N))
    sc = W.SimCfg(n_classes=4, ttft_slo_us=(10**3, 10**6, 10**9, 10**12), tpot_slo_us=(1, 5, 10, 10**9))
    met, p99 = _goodput(ctr, sc, to_dev(trh), R, 1, N, torch.from_numpy(tf).cuda(), torch.from_numpy(td).cuda())
    for r in range(R):
        row = {k: v[r] for k, v in trh.items()}
        assert (met[r], p99[r]) == orc.goodput(sc, row, tf[r], td[r]), (crowd, r)


def test_goodput_empty(orc):
    ctr = need_gpu()
    tr = ctr.empty_requests(2, 0, "cuda")
    z = torch.empty((2, 0), dtype=torch.int64, device="cuda")
    met, p99 = _goodput(ctr, W.SimCfg(), tr, 2, 1, 0, z, z)
    assert met.tolist() == [0, 0] and p99.tolist() == [-1, -1]


@pytest.mark.parametrize("wl,R,N,sets", [(W.replica_sweep(), 6, 4000, 1), (W.large_pool(rate_mreq=34_000), 2, 3000, 1),
                                         (W.replica_sweep(), 3, 45_000, 1), (W.replica_sweep(), 2, 1500, 3)])
def test_goodput_inside_simulate_matches_the_standalone_call(orc, wl, R, N, sets):
    """ctr_simulate with goodput outputs completes each row's checksum and
    computes its goodput in one pass over the outputs: the hashes equal those
    of the plain call (and the oracle's), and met / P99 equal ctr_goodput's
    and the oracle's; failed rows (a tiny FIFO) keep the checksum 0."""
    ctr = need_gpu()
    tr = gen(ctr, wl.trace, R, N)
    pols = list(W.ALL_POLICIES)
    cs = (list(W.mispriced_sets())[:sets] if sets > 1 else [wl.consts[0]])
    plain = simulate(ctr, wl.sim, cs, pols, tr, R, N)
    rows = R * len(cs) * len(pols)
    out = {k: torch.full((rows, N), -7, dtype=torch.int64, device="cuda") for k in ("tf", "td")}
    h = torch.zeros(rows, dtype=torch.int64, device="cuda")
    st = torch.full((rows,), 99, dtype=torch.int32, device="cuda")
    met = torch.full((rows,), -5, dtype=torch.int64, device="cuda")
    p99 = torch.full((rows,), -5, dtype=torch.int64, device="cuda")
    ws = ctr.simulate_workspace(wl.sim, rows, N, "cuda")
    ctr.ctr_simulate(wl.sim, cs, pols, tr, R, N, out["tf"], out["td"], h, st, ws, met_count=met, p99_ttft_us=p99)
    torch.cuda.synchronize()
    assert np.array_equal(st.cpu().numpy(), plain["status"])
    assert np.array_equal(h.cpu().numpy().astype(np.uint64), plain["hash"])
    m_alone, p_alone = _goodput(ctr, wl.sim, tr, R, len(cs) * len(pols), N, out["tf"], out["td"])
    assert np.array_equal(met.cpu().numpy(), m_alone) and np.array_equal(p99.cpu().numpy(), p_alone)
    r0 = host_trace(tr, 0)
    for j, pol in enumerate(pols):
        o = orc.simulate(wl.sim, cs[0], pol, r0)
        assert int(h[j]) & 0xFFFFFFFFFFFFFFFF == o["hash"]
        assert (int(met[j]), int(p99[j])) == orc.goodput(wl.sim, r0, o["t_first_us"], o["t_done_us"])
    # failed rows: the checksum stays 0 whichever pass completes it
    small = wl.sim.replace(cap_waiting=2, cap_pending=2)
    ctr.ctr_simulate(small, cs, pols, tr, R, N, out["tf"], out["td"], h, st, ws, met_count=met, p99_ttft_us=p99)
    torch.cuda.synchronize()
    bad = st.cpu().numpy() != 0
    assert bad.any() and not h.cpu().numpy()[bad].any()


def test_goodput_outputs_come_in_pairs():
    ctr = need_gpu()
    wl = W.replica_sweep()
    tr = gen(ctr, wl.trace, 1, 10)
    z = torch.zeros((4, 10), dtype=torch.int64, device="cuda")
    ws = ctr.simulate_workspace(wl.sim, 4, 10, "cuda")
    with pytest.raises(ctr.CtrError) as err:
        ctr.ctr_simulate(wl.sim, [W.CALIBRATED], list(W.ALL_POLICIES), tr, 1, 10, z, z.clone(),
                         torch.zeros(4, dtype=torch.int64, device="cuda"), torch.zeros(4, dtype=torch.int32,
                                                                                       device="cuda"), ws,
                         met_count=torch.zeros(4, dtype=torch.int64, device="cuda"))
    assert err.value.code == ctr.CTR_EINVAL


def _p99_tpot(ctr, sc, tr, R, rows_per, N, tf, td):
    rows = R * rows_per
    met = torch.empty(rows, dtype=torch.int64, device="cuda")
    p99 = torch.empty(rows, dtype=torch.int64, device="cuda")
    tpot = torch.full((rows,), -5, dtype=torch.int64, device="cuda")
    ctr.ctr_goodput(sc, tr, R, rows_per, N, tf, td, met, p99, p99_tpot_us=tpot)
    torch.cuda.synchronize()
    return tpot.cpu().numpy()


@pytest.mark.parametrize("wl,R,N", [(W.single_replica(), 1, 2000), (W.replica_sweep(), 8, 5000),
                                    (W.large_pool(rate_mreq=34_000), 2, 3000), (W.replica_sweep(), 3, 37),
                                    (W.document(rate_mreq=9_000), 2, 3000), (W.replica_sweep(), 1, 45_000)])
def test_p99_tpot_matches_oracle(orc, wl, R, N):
    """Table 2's P99 TPOT of every simulated row, bit for bit."""
    ctr = need_gpu()
    tr = gen(ctr, wl.trace, R, N)
    pols = list(W.ALL_POLICIES)
    res = simulate(ctr, wl.sim, [wl.consts[0]], pols, tr, R, N)
    tpot = _p99_tpot(ctr, wl.sim, tr, R, len(pols), N, torch.from_numpy(res["t_first_us"]).cuda(),
                     torch.from_numpy(res["t_done_us"]).cuda())
    for r in range(R):
        trh = host_trace(tr, r)
        for j in range(len(pols)):
            row = r * len(pols) + j
            assert tpot[row] == orc.p99_tpot(trh, res["t_first_us"][row], res["t_done_us"][row]), (r, j)


@pytest.mark.parametrize("case", ["crowded", "wide", "negative", "one_token", "few", "empty"])
def test_p99_tpot_adversarial(orc, case):
    """Crowded bins (over 512 equal TPOTs at the rank), decode times of 2^32 us and more, negative
    decode times (radix select), rows without a multi-token request (-1), single requests, empty rows."""
    ctr = need_gpu()
    rng = np.random.default_rng(len(case))
    R, N = 3, 6000
    o = rng.integers(1, 300, (R, N))
    o[rng.random((R, N)) < 0.2] = 1
    tf = rng.integers(0, 10**9, (R, N))
    td = tf + rng.integers(0, 10**7, (R, N))
    if case == "crowded":
        td = tf + 30_000 * np.maximum(o - 1, 0) + rng.integers(0, 2, (R, N))  # TPOTs 30,000 or just above
    elif case == "wide":
        td[:, 5] = tf[:, 5] + (1 << 33) + 12345
    elif case == "negative":
        td[1] = tf[1] - rng.integers(0, 10**6, N)
    elif case == "one_token":
        o[:] = 1
    elif case == "few":
        o[:] = 1
        o[0, 17] = 2
        o[2, :3] = 7
    elif case == "empty":
        N = 0
        o, tf, td = o[:, :0], tf[:, :0], td[:, :0]
    trh = {"arrival_us": np.sort(rng.integers(0, 10**6, (R, N)), axis=1), "prompt_len": np.ones((R, N)),
           "true_out": o, "pred_out": np.ones((R, N)), "slo_class": np.zeros((R, N))}
    tpot = _p99_tpot(ctr, W.SimCfg(), to_dev(trh), R, 1, N, torch.from_numpy(tf).cuda(), torch.from_numpy(td).cuda())
    for r in range(R):
        assert tpot[r] == orc.p99_tpot({"true_out": o[r]}, tf[r], td[r]), (case, r)
    if case in ("one_token", "empty"):
        assert tpot.tolist() == [-1, -1, -1]
