"""Failure handling with a live GPU: injected allocation failure, freed handles,
argument errors, a non-finite weight latched on the device and reported by
mone_mem_sync, and a bounded device wait that runs out.  Nothing here faults or
hangs the GPU: every failure is made on the host, by the data, or by a wait with
a 1 ms limit on a barrier that no copy will complete (nothing is in flight when it
gives up)."""
import math
import os
import time

import pytest
import torch

import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import DeviceRun, config_of, oracle_chain, rel_fro

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def small(mode=wk.PLAIN, dtype="bf16"):
    return wk.Workload(f"fault_{dtype}", 40 + mode, 1, 2, 256, 256, 256, 2, 64, 256, 512, 16, dtype, mode, 0.1)


def code_of(fn, *a, **k):
    with pytest.raises(mone.MoneError) as ei:
        fn(*a, **k)
    return ei.value.code


def test_injected_allocation_failure_reports_oom_and_leaks_nothing():
    wl = small()
    W1, W2 = wk.initial_weights(wl, "cuda")
    os.environ["MONE_FAULT_ALLOC"] = "1"
    try:
        assert code_of(mone.mone_mem_init, config_of(wl), W1, W2) == 3
    finally:
        del os.environ["MONE_FAULT_ALLOC"]
    h = mone.mone_mem_init(config_of(wl), W1, W2)
    mone.mone_mem_free(h)


def test_freed_handle_is_rejected():
    wl = small()
    run = DeviceRun(wl)
    h = run.h
    mone.mone_mem_free(h)
    run.h = None
    assert code_of(mone.mone_mem_free, h) == 1
    assert code_of(mone.mone_ttl_context, h, run.X, run.K, run.V, wl.N) == 1
    assert mone.mone_mem_launch_count(h) == -1


def test_argument_errors_launch_nothing():
    wl = small()
    run = DeviceRun(wl)
    before = mone.mone_mem_launch_count(run.h)
    x = run.X[0, 0]
    assert code_of(mone.mone_ttl_segment, run.h, 0, 0, x, run.K[0, 0], run.V[0, 0], wl.seg_T + 1) == 1
    assert code_of(mone.mone_ttl_segment, run.h, 1, 0, x, run.K[0, 0], run.V[0, 0], 8) == 1
    assert code_of(mone.mone_ttl_segment, run.h, 0, 5, x, run.K[0, 0], run.V[0, 0], 8) == 1
    assert code_of(mone.mone_ttl_segment, run.h, 0, 0, x.data_ptr() + 2, run.K[0, 0], run.V[0, 0], 8) == 1
    assert code_of(mone.mone_ttl_context, run.h, run.X, run.K, run.V, 0) == 1
    Xq = wk.query_inputs(wl, "cuda")
    Ko = torch.empty(1, 2, 2, 16, 64, dtype=torch.bfloat16, device="cuda")
    assert code_of(mone.mone_mem_generate_kv, run.h, Xq, 0, Ko, Ko, (0, 0, 0, 0)) == 1
    assert code_of(mone.mone_mem_generate_kv, run.h, Xq, 16, Ko, Ko, (-1, 0, 0, 0)) == 1
    seg = torch.zeros(8, wl.chains, device="cuda")
    assert code_of(mone.mone_ttl_context_metrics, run.h, run.X, run.K, run.V, wl.N, seg.data_ptr() + 2, None) == 1
    assert code_of(mone.mone_ttl_context_metrics, run.h, run.X, run.K, run.V, wl.N, None, seg.data_ptr() + 1) == 1
    assert code_of(mone.mone_ttl_context_metrics, run.h, run.X, run.K, run.V, 0, seg, seg) == 1
    assert mone.mone_mem_launch_count(run.h) == before
    run.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_nonfinite_weight_is_latched_and_the_handle_recovers(dtype):
    wl = small(dtype=dtype)
    run = DeviceRun(wl)
    X = run.X.clone()
    X[0, 1, 3, 5] = float("nan")
    mone.mone_ttl_context(run.h, X, run.K, run.V, wl.N)
    assert code_of(mone.mone_mem_sync, run.h) == 6
    mone.mone_mem_sync(run.h)  # the latch is cleared once reported
    # the handle stays usable: reset the state and learn from clean inputs
    mone.mone_mem_write_state(run.h, run.W1_0, run.W2_0)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    assert bool(torch.isfinite(W1).all()) and bool(torch.isfinite(W2).all())
    run.close()


@pytest.mark.parametrize("T", [256, 128])  # phase A on CTA pairs (T / 128 even), and the one-CTA kernel
def test_bounded_wait_runs_out_and_the_handle_recovers(T):
    # MONE_FAULT_STALL=1 at init: the handle's first tensor-core phase-A launch issues no loads
    # and gives every wait 1 ms.  Its MMA issuer's first wait for a full stage runs out (no copy
    # and no MMA has been issued), the epilogue warps' waits for the accumulator run out too,
    # every role reaches the kernel's final barrier, TMEM is released, and DEV_TIMEOUT is
    # latched; mone_mem_sync reports MONE_ERR_TIMEOUT.
    wl = wk.Workload(f"fault_stall_{T}", 45, 1, 2, 256, 256, 256, 2, 64, T, 2 * T, 16, "bf16", wk.PLAIN, 0.1)
    os.environ["MONE_FAULT_STALL"] = "1"
    try:
        run = DeviceRun(wl)
    finally:
        del os.environ["MONE_FAULT_STALL"]
    t0 = time.time()
    mone.mone_ttl_context(run.h, run.X, run.K, run.V, wl.N)
    assert code_of(mone.mone_mem_sync, run.h) == 5  # MONE_ERR_TIMEOUT
    assert time.time() - t0 < 1.5                  # the launch's 1 ms limit, not the default 2 s
    mone.mone_mem_sync(run.h)                      # the latch is cleared once reported
    # the handle stays usable: reset the state, learn the whole context again, match the oracle
    mone.mone_mem_write_state(run.h, run.W1_0, run.W2_0)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    for c in range(wl.chains):
        st, _ = oracle_chain(run, c)
        assert rel_fro(W1[c], st.W["W1"]) <= 2e-2 and rel_fro(W2[c], st.W["W2"]) <= 2e-2, c
    run.close()
