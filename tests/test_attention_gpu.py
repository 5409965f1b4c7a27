"""GPU parity of the consumer attention (Eq. 5, reading R14) against the oracle's definition.

The caches hold memory tokens at positions [0, n_mem) and the query tokens' own keys and
values after them.  Where the case says so, the memory tokens are the library's own read
(mone_mem_generate_kv after a test-time-learning pass); otherwise they are random.
Tolerances: bf16 path 1e-2 (outputs rounded to bf16, fp32 accumulation), fp32 path 1e-5.
bf16 caches whose rows are 16-byte aligned take the tensor-core kernel (keys in chunks of 256
positions); other bf16 layouts and fp32 take the CUDA-core kernel.  Both are covered here.
"""
import pytest
import torch

import oracle as O
import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import DeviceRun, rel_fro

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    mone.lib()


def small(mode=wk.PAPER, dtype="bf16", n_ctx=1, n_layers=2, d_out=256, hd=64, N=600, Q=40):
    return wk.Workload(f"attn_{dtype}", 40, n_ctx, n_layers, 256, 256, d_out, d_out // (2 * hd), hd, 256 if dtype ==
                       "bf16" else 128, N, Q, dtype, mode, 0.3 if dtype == "bf16" else 1e-2)


def run_case(wl, n_q, Lq, n_mem, seed, memory_from_read=True, pos_pad=0):
    """pos_pad: extra elements after each cache position (a position stride of head_dim + pos_pad)."""
    run = DeviceRun(wl)
    run.ttl_context()
    dt = wl.torch_dtype()
    g = torch.Generator(device="cuda").manual_seed(seed)
    S = n_mem + Lq + 3  # spare positions at the end: the kernel must not read them
    shape = (wl.n_ctx, wl.n_layers, wl.n_kv_heads, S, wl.head_dim + pos_pad)
    Kc = torch.randn(*shape, generator=g, device="cuda").to(dt)[..., :wl.head_dim]
    Vc = torch.randn(*shape, generator=g, device="cuda").to(dt)[..., :wl.head_dim]
    strides = Kc.stride()[:4]
    if memory_from_read and n_mem:
        Xq = wk.query_inputs(wl, "cuda", Q=n_mem)
        mone.mone_mem_generate_kv(run.h, Xq, n_mem, Kc, Vc, strides)
    Qt = torch.randn(wl.n_ctx, wl.n_layers, n_q, Lq, wl.head_dim, generator=g, device="cuda").to(dt)
    out = torch.full_like(Qt, 7.0)
    mone.mone_attention(run.h, Qt, n_q, Lq, Kc, Vc, strides, n_mem, out)
    mone.mone_mem_sync(run.h)
    run.close()
    return Qt.cpu(), Kc.cpu(), Vc.cpu(), out.cpu()


def check(wl, Qt, Kc, Vc, out, n_mem, Lq, tol):
    for ctx in range(wl.n_ctx):
        for layer in range(wl.n_layers):
            ref = O.attention(Qt[ctx, layer], Kc[ctx, layer, :, :n_mem + Lq], Vc[ctx, layer, :, :n_mem + Lq], n_mem)
            assert rel_fro(out[ctx, layer].float(), ref) <= tol, (ctx, layer)


@pytest.mark.parametrize("group,Lq,n_mem", [
    (2, 40, 40),      # query heads in pairs, memory = the read of 40 query tokens
    (1, 70, 0),       # no memory: causal self-attention; 70 tokens = two tiles, the last ragged
    (7, 20, 150),     # 7 heads per KV head (tiles of 9 tokens), memory over three 64-position chunks
    (2, 1, 300),      # one decode token over a long memory: two key chunks on the tensor cores
    (1, 130, 400),    # 128-token tiles, the second ragged; up to 530 keys = three chunks
    (64, 5, 10),      # the largest group: 2 tokens x 64 heads per 128-row tile
])
def test_attention_bf16(group, Lq, n_mem):
    wl = small(n_ctx=2)
    n_q = group * wl.n_kv_heads
    Qt, Kc, Vc, out = run_case(wl, n_q, Lq, n_mem, seed=group * 100 + Lq)
    check(wl, Qt, Kc, Vc, out, n_mem, Lq, 1e-2)


@pytest.mark.parametrize("group,Lq,n_mem", [(2, 40, 40), (3, 9, 70)])
def test_attention_bf16_unaligned_cache_rows(group, Lq, n_mem):
    """Position stride head_dim + 4 (8 bytes past a 16-byte multiple): the CUDA-core kernel."""
    wl = small()
    Qt, Kc, Vc, out = run_case(wl, group * wl.n_kv_heads, Lq, n_mem, seed=31 + group, pos_pad=4)
    check(wl, Qt, Kc, Vc, out, n_mem, Lq, 1e-2)


@pytest.mark.parametrize("Lq,n_mem", [
    (33, 77),    # one key chunk
    (5, 400),    # two key chunks: at hd 128 the probabilities take the key buffer, restaged per chunk
])
def test_attention_bf16_head_dim_128_random_memory(Lq, n_mem):
    wl = small(d_out=512, hd=128)
    Qt, Kc, Vc, out = run_case(wl, 3 * wl.n_kv_heads, Lq, n_mem, seed=5 + n_mem, memory_from_read=False)
    check(wl, Qt, Kc, Vc, out, n_mem, Lq, 1e-2)


def test_attention_at_the_bench_shape():
    """The shape bench.py times: 16 chains (one context, 16 layers), 8 KV heads x 2 query heads,
    hd 64, 64 memory tokens from the read plus 64 query tokens; every chain checked."""
    wl = small(n_ctx=1, n_layers=16, d_out=1024, hd=64, N=256, Q=64)
    Qt, Kc, Vc, out = run_case(wl, 2 * wl.n_kv_heads, 64, 64, seed=77)
    check(wl, Qt, Kc, Vc, out, 64, 64, 1e-2)


def test_attention_fp32():
    wl = small(mode=wk.PLAIN, dtype="f32", N=300, Q=32)
    Qt, Kc, Vc, out = run_case(wl, 2 * wl.n_kv_heads, 33, 32, seed=9)
    check(wl, Qt, Kc, Vc, out, 32, 33, 1e-5)


def test_attention_argument_errors_launch_nothing():
    wl = small()
    run = DeviceRun(wl)
    Kc = torch.zeros(1, 2, wl.n_kv_heads, 16, wl.head_dim, dtype=torch.bfloat16, device="cuda")
    Qt = torch.zeros(1, 2, 2 * wl.n_kv_heads, 4, wl.head_dim, dtype=torch.bfloat16, device="cuda")
    st = Kc.stride()[:4]
    n0 = mone.mone_mem_launch_count(run.h)
    bad = [
        (3, 4, st, 0),                       # query heads not a multiple of the KV heads
        (2 * wl.n_kv_heads, 0, st, 0),       # no query tokens
        (2 * wl.n_kv_heads, 4, st, -1),      # negative memory length
        (2 * wl.n_kv_heads, 4, (st[0], st[1], st[2], -st[3]), 0),  # negative stride
        (2 * wl.n_kv_heads, 4, (st[0], st[1], st[2], 8), 0),       # positions overlap within a head
    ]
    for n_q, Lq, strides, n_mem in bad:
        with pytest.raises(mone.MoneError) as e:
            mone.mone_attention(run.h, Qt, n_q, Lq, Kc, Kc, strides, n_mem, Qt)
        assert e.value.code == 1
    assert mone.mone_mem_launch_count(run.h) == n0
    run.close()
