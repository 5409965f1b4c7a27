"""The allocation-free memory read, checked against the ordinary one.

Some callers cannot allocate device memory while they serve queries: a
framework whose caching allocator already holds the GPU's free memory, or a
serving loop that cannot afford cudaMalloc's device synchronisation.  For them
the library offers mone_mem_generate_kv_noalloc, which reads the memory through
a fixed scratch array compiled into the library instead of allocating one.
This file runs last so that a failure here leaves every other test's result
intact; it also passes when run alone in a fresh process.
"""
import ctypes

import pytest
import torch

import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import DeviceRun

pytestmark = pytest.mark.gpu

@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def outputs(wl, Q, dtype):
    K = torch.empty(wl.n_ctx, wl.n_layers, wl.n_kv_heads, Q, wl.head_dim, dtype=dtype, device="cuda")
    return K, torch.empty_like(K)


@pytest.mark.parametrize("dtype,mode,hd,strided", [("bf16", wk.PAPER, 64, False), ("f32", wk.PLAIN, 64, False),
                                                    ("bf16", wk.PAPER, 128, False), ("bf16", wk.PLAIN, 64, True),
                                                    ("f32", wk.PAPER, 128, True)])
def test_noalloc_read_matches_the_allocating_read_twice(dtype, mode, hd, strided):
    # the same kernels on the same inputs, only the scratch differs: the outputs agree bit for bit,
    # on two calls in a row (the second one reads what the first left in the shared array)
    wl = wk.Workload(f"noalloc_{dtype}", 30 + mode, 2, 2, 256, 256, 256, 256 // (2 * hd), hd, 256, 512 + 77, 40,
                     dtype, mode, 0.3)
    run = DeviceRun(wl)
    run.ttl_context()
    Xq = wk.query_inputs(wl, "cuda")
    strides = mone.kv_strides(wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim)
    Kref, Vref = outputs(wl, wl.Q, Xq.dtype)
    mone.mone_mem_generate_kv(run.h, Xq, wl.Q, Kref, Vref, strides)
    mone.mone_mem_sync(run.h)
    off, S_tot = 5, wl.Q + 11       # strided: the memory tokens land inside a longer attention cache
    for _ in range(2):
        if strided:
            ck = torch.full((wl.n_ctx, wl.n_layers, wl.n_kv_heads, S_tot, wl.head_dim), 3.0, dtype=Xq.dtype,
                            device="cuda")
            cv = ck.clone()
            mone.mone_mem_generate_kv_noalloc(run.h, Xq, wl.Q, ck[:, :, :, off:], cv[:, :, :, off:], ck.stride()[:4])
            mone.mone_mem_sync(run.h)
            K, V = ck[:, :, :, off:off + wl.Q], cv[:, :, :, off:off + wl.Q]
            assert bool((ck[:, :, :, :off] == 3).all()) and bool((ck[:, :, :, off + wl.Q:] == 3).all())
            assert bool((cv[:, :, :, :off] == 3).all()) and bool((cv[:, :, :, off + wl.Q:] == 3).all())
        else:
            K, V = outputs(wl, wl.Q, Xq.dtype)
            mone.mone_mem_generate_kv_noalloc(run.h, Xq, wl.Q, K, V, strides)
            mone.mone_mem_sync(run.h)
        assert torch.equal(K, Kref) and torch.equal(V, Vref)
    run.close()


def test_noalloc_read_refuses_the_swiglu_memory_before_any_work():
    wl = wk.Workload("noalloc_sw", 33, 1, 2, 256, 96, 256, 2, 64, 128, 128, 16, "bf16", wk.PAPER, 0.3,
                     memory="swiglu", heads=2)
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    Xq = wk.query_inputs(wl, "cuda")
    K, V = outputs(wl, wl.Q, Xq.dtype)
    arr = (ctypes.c_longlong * 4)(*mone.kv_strides(wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim))
    before = mone.mone_mem_launch_count(run.h)
    rc = mone.lib().mone_mem_generate_kv_noalloc(run.h, Xq.data_ptr(), wl.Q, K.data_ptr(), V.data_ptr(), arr,
                                                 torch.cuda.current_stream().cuda_stream)
    assert rc == 7  # MONE_ERR_UNSUPPORTED
    assert "SwiGLU" in mone.mone_last_error()
    assert mone.mone_mem_launch_count(run.h) == before
    mone.mone_mem_sync(run.h)
    run.close()


def test_noalloc_read_rejects_work_beyond_its_scratch():
    wl = wk.Workload("noalloc_big", 32, 1, 4, 256, 256, 256, 2, 64, 256, 256, 4096, "bf16", wk.PLAIN, 0.3)
    run = DeviceRun(wl)
    Xq = torch.zeros(wl.n_ctx, wl.n_layers, wl.Q, wl.d_in, dtype=torch.bfloat16, device="cuda")
    K, V = outputs(wl, wl.Q, Xq.dtype)
    arr = (ctypes.c_longlong * 4)(*mone.kv_strides(wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim))
    rc = mone.lib().mone_mem_generate_kv_noalloc(run.h, Xq.data_ptr(), wl.Q, K.data_ptr(), V.data_ptr(), arr,
                                                 torch.cuda.current_stream().cuda_stream)
    assert rc == 2  # MONE_ERR_UNSUPPORTED_SHAPE, before any GPU work
    assert "exceeds the fixed scratch" in mone.mone_last_error()
    mone.mone_mem_sync(run.h)
    run.close()
