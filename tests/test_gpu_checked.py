"""The simulator's and the goodput pass's parity cases again, on
libctr_checked.so: the same kernels compiled with CTR_BOUNDS_CHECK=1, so that
every index into the workspace (heaps, rings, FIFOs), the trace, the outputs
and goodput's shared histograms, staged bins and P99 candidates is compared
with its buffer's length before the access.  An index outside would skip the
access and end its row with CTR_EBOUNDS (in the simulator's status, in
goodput's met count and P99), which no oracle value equals, so each case below
passes only if no access of the run left its buffer.  This is the device-side
memory check where no memory checker runs: tiny capacities (every overflow
path), every pool width, batched prefill, the proxy's signals, random
configurations, adversarial and crowded TTFTs, and the benchmarked launch."""
import pytest
import torch

import simutil as U
import test_gpu_fuzz as F
import test_gpu_goodput as G
import test_gpu_sim as S
from gpuutil import need_gpu
from paper_2609_16206_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def checked_library():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16206_gb300 import build, ctr
    build.build()
    path = build.build(checked=True)
    before = ctr.use_library(path)
    yield ctr
    ctr.use_library(before)


def test_is_the_checked_build():
    ctr = need_gpu()
    assert ctr.ctr_bounds_checked() == 1


@pytest.mark.parametrize("case", U.worked_traces(), ids=lambda c: c["name"])
def test_worked_traces(orc, case):
    S.test_worked_traces(orc, case)


@pytest.mark.parametrize("n_pre,n_dec", [(1, 1), (31, 1), (1, 31), (3, 5)])
def test_pool_shapes(orc, n_pre, n_dec):
    S.test_pool_shapes(orc, n_pre, n_dec)


@pytest.mark.parametrize("N", [0, 1, 33])
def test_ragged_and_empty(orc, N):
    S.test_ragged_and_empty(orc, N)


def test_small_workspace(orc):
    S.test_small_workspace_same_results(orc)


def test_capacity_overflow(orc):
    S.test_capacity_overflow_matches_oracle(orc)


def test_step_budget_and_invalid_rows(orc):
    S.test_step_budget_and_invalid_rows(orc)


@pytest.mark.parametrize("caps", [dict(cap_prefill_ring=24), dict(cap_pending=12), dict(cap_waiting=2),
                                  dict(cap_active=20)], ids=lambda c: list(c)[0])
def test_batched_prefill_capacity_errors(orc, caps):
    S.test_batched_prefill_capacity_errors(orc, caps)


@pytest.mark.parametrize("wl", [W.replica_sweep(), W.large_pool(rate_mreq=34_000)], ids=["2p6d", "4p28d"])
def test_proxy_signals(orc, wl):
    S.test_proxy_signals(orc, wl)


@pytest.mark.parametrize("wl", [W.replica_sweep(), W.large_pool(rate_mreq=34_000)], ids=["2p6d", "4p28d"])
def test_power_of_two_router(orc, wl):
    S.test_power_of_two_router(orc, wl)


@pytest.mark.parametrize("budget", [900, 1 << 20])
def test_batched_prefill_document(orc, budget):
    S.test_batched_prefill_document(orc, budget)


@pytest.mark.parametrize("seed", range(0, 160, 4))
def test_random_configuration(orc, seed):
    F.test_random_configuration(orc, seed)


@pytest.mark.parametrize("wl,R,N", [(W.replica_sweep(), 8, 5000), (W.large_pool(rate_mreq=34_000), 2, 3000),
                                    (W.replica_sweep(), 3, 37), (W.replica_sweep(), 1, 45_000)],
                         ids=["2p6d", "4p28d", "short", "unstaged"])
def test_goodput(orc, wl, R, N):
    G.test_goodput_matches_oracle(orc, wl, R, N)


def test_goodput_adversarial_times(orc):
    G.test_goodput_adversarial_times(orc)


@pytest.mark.parametrize("crowd", [1, 512, 513, 3000])
def test_goodput_crowded_p99_bin(orc, crowd):
    G.test_goodput_crowded_p99_bin(orc, crowd)


@pytest.mark.parametrize("wl,R,N,sets", [(W.replica_sweep(), 6, 4000, 1), (W.replica_sweep(), 3, 45_000, 1)],
                         ids=["staged", "unstaged"])
def test_goodput_inside_simulate(orc, wl, R, N, sets):
    G.test_goodput_inside_simulate_matches_the_standalone_call(orc, wl, R, N, sets)


def test_benchmarked_launch(orc):
    """4,096 bursty replicas x 20,000 requests x 4 policies in one launch: every row OK (no CTR_EBOUNDS),
    sampled rows equal to the oracle."""
    S.test_full_size_sweep_sampled(orc)
