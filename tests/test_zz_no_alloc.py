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
from harness import DeviceRun, rel_fro

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def outputs(wl, Q, dtype):
    K = torch.empty(wl.n_ctx, wl.n_layers, wl.n_kv_heads, Q, wl.head_dim, dtype=dtype, device="cuda")
    return K, torch.empty_like(K)


@pytest.mark.parametrize("dtype,mode", [("bf16", wk.PAPER), ("f32", wk.PLAIN)])
def test_noalloc_read_matches_the_allocating_read_twice(dtype, mode):
    wl = wk.Workload(f"noalloc_{dtype}", 30 + mode, 2, 2, 256, 256, 256, 2, 64, 256, 512 + 77, 40, dtype, mode, 0.3)
    run = DeviceRun(wl)
    run.ttl_context()
    Xq = wk.query_inputs(wl, "cuda")
    strides = mone.kv_strides(wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim)
    Kref, Vref = outputs(wl, wl.Q, Xq.dtype)
    mone.mone_mem_generate_kv(run.h, Xq, wl.Q, Kref, Vref, strides)
    mone.mone_mem_sync(run.h)
    for _ in range(2):
        K, V = outputs(wl, wl.Q, Xq.dtype)
        mone.mone_mem_generate_kv_noalloc(run.h, Xq, wl.Q, K, V, strides)
        mone.mone_mem_sync(run.h)
        assert rel_fro(K.float().cpu(), Kref.float().cpu()) <= TOL[dtype]
        assert rel_fro(V.float().cpu(), Vref.float().cpu()) <= TOL[dtype]
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
