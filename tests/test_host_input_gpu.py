"""GPU: test-time learning of a context held in host memory (mone_ttl_context_host).

The library gathers chunks of whole segments from host memory into its device windows and
learns each chunk with the call mone_ttl_context makes.  So the result must equal
mone_ttl_context called on the same chunks from device memory, and the state must match the
oracle's chain (Eq. 9) within the path's tolerance (bf16 2e-2, fp32 1e-4; see test_parity_gpu).

"Equal" is bit for bit where the learning is deterministic: plain mode and the fp32 resident
kernel.  With row renormalisation (paper mode) on the bf16 (MLP and SwiGLU) and fp32 tiled paths, phase B adds a
row's sum of squares from its column tiles with float atomics, so two runs of the same call
differ in the last bits of the renormalisation scale; there the bound is relative (bf16 1e-3,
the bound of the split-context test, which also covers bf16 rounding flips that such a bit
can cause; fp32 1e-5).
"""
import pytest
import torch

import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import DeviceRun, oracle_read, rel_fro
from test_parity_gpu import BF16_TOL, F32_TOL, check_chain, small
from test_swiglu_gpu import check as check_swiglu, swiglu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    mone.lib()


def pinned(t):
    h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
    h.copy_(t)
    return h


def device_chunks(run, bounds):
    """mone_ttl_context on device copies of the chunks (r0, n) in order (an int: chunks of that length)."""
    if isinstance(bounds, int):
        bounds = [(r0, min(bounds, run.N - r0)) for r0 in range(0, run.N, bounds)]
    for r0, nr in bounds:
        X, K, V = (t[:, :, r0:r0 + nr].contiguous() for t in (run.X, run.K, run.V))
        mone.mone_ttl_context(run.h, X, K, V, nr)
    mone.mone_mem_sync(run.h)


def assert_same_state(a, b, tol=0.0):
    for ta, tb in zip(a.state(), b.state()):
        if tol == 0.0:
            assert torch.equal(ta, tb)
        else:
            assert rel_fro(ta, tb) <= tol


CASES = [
    # (workload, chunk tokens, host-vs-device bound): ragged last chunks, the library's own
    # chunk length (one chunk here), plain mode, the fp32 tiled path and the fp32 resident path
    ("bf16_paper", 2 * 256, 1e-3),
    ("bf16_paper", 0, 1e-3),
    ("bf16_plain", 0, 0.0),
    ("bf16_plain", 256, 0.0),
    ("f32_tiled", 3 * 64, 1e-5),
    ("f32_resident", 3 * 128, 0.0),
    ("swiglu", 2 * 256, 1e-3),
]


def workload(name):
    if name == "bf16_paper":
        return small(wk.PAPER)
    if name == "bf16_plain":
        return small(wk.PLAIN)
    if name == "f32_tiled":
        return small(wk.PAPER, "f32", n_ctx=1, T=64, N=7 * 64 + 20, d_in=512, d_hid=128, d_out=256, lr=0.5)
    if name == "swiglu":  # the per-head SwiGLU of Eq. 3: 2 heads of 128, ragged hidden tiles (96 units)
        return swiglu(T=256, N=4 * 256 + 37)
    return wk.WORKLOADS["tiny_f32"]


@pytest.mark.parametrize("name,chunk,same", CASES)
def test_host_context_equals_device_chunks_and_the_oracle(name, chunk, same):
    wl = workload(name)
    a = DeviceRun(wl)
    hX, hK, hV = pinned(a.X), pinned(a.K), pinned(a.V)
    mone.mone_mem_set_timing(a.h, 1)
    mone.mone_ttl_context_host(a.h, hX, hK, hV, a.N, chunk)
    mone.mone_mem_sync(a.h)
    ct = chunk if chunk else -(-a.N // wl.seg_T) * wl.seg_T  # this workload: the library takes one chunk
    assert mone.mone_mem_kernel_time(a.h, mone.KERNEL_KINDS.index("stage"))[1] == -(-a.N // ct)
    b = DeviceRun(wl)
    device_chunks(b, ct)
    assert_same_state(a, b, same)
    if wl.memory == "swiglu":
        check_swiglu(a, range(wl.chains))
    else:
        W1, W2, _, _ = a.state()
        tol = F32_TOL if wl.dtype == "f32" else BF16_TOL
        for c in range(wl.chains):
            check_chain(a, c, W1, W2, tol)
    a.close()
    b.close()


def test_host_context_continues_the_state_across_calls():
    # two host calls (the first a whole number of segments) equal the same two calls from device
    wl = small(wk.PLAIN)
    a, b = DeviceRun(wl), DeviceRun(wl)
    n1 = 2 * wl.seg_T
    parts = [(slice(0, n1), n1), (slice(n1, a.N), a.N - n1)]
    for sl, n in parts:
        hX, hK, hV = (pinned(t[:, :, sl].contiguous()) for t in (a.X, a.K, a.V))
        mone.mone_ttl_context_host(a.h, hX, hK, hV, n, wl.seg_T)
        mone.mone_mem_sync(a.h)  # the host tensors of this part are released after the call
        X, K, V = (t[:, :, sl].contiguous() for t in (b.X, b.K, b.V))
        for r0 in range(0, n, wl.seg_T):
            nr = min(wl.seg_T, n - r0)
            mone.mone_ttl_context(b.h, X[:, :, r0:r0 + nr].contiguous(), K[:, :, r0:r0 + nr].contiguous(),
                                  V[:, :, r0:r0 + nr].contiguous(), nr)
    mone.mone_mem_sync(b.h)
    assert_same_state(a, b)
    a.close()
    b.close()


def test_host_context_from_pageable_memory():
    # where the device reads host memory through the host's page tables (Grace), ordinary
    # pageable memory is accepted; elsewhere the call refuses it before any work
    wl = small(wk.PLAIN)
    a, b = DeviceRun(wl), DeviceRun(wl)
    hX, hK, hV = (t.cpu() for t in (a.X, a.K, a.V))
    assert not hX.is_pinned()
    n0 = mone.mone_mem_launch_count(a.h)
    try:
        mone.mone_ttl_context_host(a.h, hX, hK, hV, a.N, 2 * wl.seg_T)
    except mone.MoneError as e:
        assert e.code == 1 and mone.mone_mem_launch_count(a.h) == n0
        pytest.skip("this device does not read pageable host memory")
    mone.mone_mem_sync(a.h)
    device_chunks(b, 2 * wl.seg_T)
    assert_same_state(a, b)
    a.close()
    b.close()


def test_host_context_argument_errors_launch_nothing():
    wl = small(wk.PAPER)
    run = DeviceRun(wl)
    hX, hK, hV = pinned(run.X), pinned(run.K), pinned(run.V)
    T = wl.seg_T
    n0 = mone.mone_mem_launch_count(run.h)
    bad = [
        ((run.X, hK, hV), run.N, 0),                 # device memory: mone_ttl_context takes it
        ((hX, hK, hV), 0, 0),                         # no tokens
        ((hX, hK, hV), run.N, T + 64),                # chunk not a whole number of segments
        ((hX, hK, hV), run.N, -T),                    # negative chunk
        ((hX.view(-1)[1:], hK, hV), run.N, 0),        # X not 16-byte aligned
    ]
    for (X, K, V), N, ct in bad:
        with pytest.raises(mone.MoneError) as e:
            mone.mone_ttl_context_host(run.h, X, K, V, N, ct)
        assert e.value.code == 1, (N, ct)
    assert mone.mone_mem_launch_count(run.h) == n0
    run.close()


def test_host_context_at_the_bench_size_sampled_chains():
    """The configuration bench.py's e2e runs: l16_d2048_128k, the 128K-token context in pinned
    host memory (8.6 GB of X: offsets past 2^31 bytes), the library's chunks (5,120 tokens, 26
    gathers) on SMs of their own.  The first and the last chain are checked against the oracle
    (state and read)."""
    wl = wk.WORKLOADS["l16_d2048_128k"]
    run = DeviceRun(wl)
    hX, hK, hV = pinned(run.X), pinned(run.K), pinned(run.V)
    mone.mone_mem_set_timing(run.h, 1)
    mone.mone_ttl_context_host(run.h, hX, hK, hV, run.N)
    mone.mone_mem_sync(run.h)
    assert mone.mone_mem_kernel_time(run.h, mone.KERNEL_KINDS.index("stage"))[1] == -(-run.N // 5120)
    mone.mone_mem_set_timing(run.h, 0)
    del hX, hK, hV
    W1, W2, _, _ = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in (0, wl.chains - 1):
        st = check_chain(run, c, W1, W2, BF16_TOL)
        Ko, Vo = oracle_read(run, st, c, Xq)
        ctx, layer = divmod(c, wl.n_layers)
        assert rel_fro(Kg[ctx, layer].float(), Ko) <= BF16_TOL
        assert rel_fro(Vg[ctx, layer].float(), Vo) <= BF16_TOL
    run.close()
    torch.cuda.empty_cache()
