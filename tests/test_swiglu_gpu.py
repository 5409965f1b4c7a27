"""GPU parity of the per-head SwiGLU memory (Eq. 3; memory = MONE_MEM_SWIGLU) against the
oracle's swiglu form.  Tolerances as for the two-matrix memory: weights and generated K/V
within 2e-2 relative Frobenius error after the whole context (bf16 operands, fp32 state),
and the weight change W_S - W_0 within the same 2e-2 (per hidden row: 8e-2)."""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import DeviceRun, gpu_layout, oracle_chain, oracle_init, oracle_read, record, rel_fro, row_rel_errors

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    mone.lib()


def swiglu(mode=wk.PAPER, n_ctx=1, n_layers=2, d=256, heads=2, F=96, n_kv=2, hd=64, T=128, N=3 * 128 + 50, Q=40,
           lr=0.3):
    return wk.Workload(f"sw_{mode}_{d}", 60 + mode, n_ctx, n_layers, d, F, d, n_kv, hd, T, N, Q, "bf16", mode, lr,
                       memory="swiglu", heads=heads)


DW_TOL = 2e-2      # the weight change W_S - W_0, as the weights
ROW_DW_TOL = 8e-2  # per hidden row, relative error of the weight change (see test_parity_gpu)


def check(run, chains, Xq=None):
    W1, W2, _, _ = run.state()
    Kg = Vg = None
    if Xq is not None:
        Kg, Vg = run.generate_kv(Xq)
    for c in chains:
        st, _ = oracle_chain(run, c)
        o1, o2 = gpu_layout(run.wl, st.W)
        e1 = record("swiglu", "W1", rel_fro(W1[c], o1), TOL)
        e2 = record("swiglu", "W2", rel_fro(W2[c], o2), TOL)
        assert e1 <= TOL and e2 <= TOL, (c, e1, e2)
        s1, s2 = gpu_layout(run.wl, oracle_init(run.wl, run.W1_0[c], run.W2_0[c]).W)
        g1, g2 = W1[c].double().numpy() - s1, W2[c].double().numpy() - s2
        d1 = record("swiglu", "dW1", rel_fro(g1, o1 - s1), DW_TOL)
        d2 = record("swiglu", "dW2", rel_fro(g2, o2 - s2), DW_TOL)
        assert d1 <= DW_TOL and d2 <= DW_TOL, (c, d1, d2)
        # rows of the library layout: W1 holds [W_in | W_gate] per hidden unit, W2 = W_out
        r1 = record("swiglu", "dW1 row", row_rel_errors(g1, o1 - s1).max(), ROW_DW_TOL)
        r2 = record("swiglu", "dW2 row", row_rel_errors(g2, o2 - s2).max(), ROW_DW_TOL)
        assert r1 <= ROW_DW_TOL and r2 <= ROW_DW_TOL, (c, r1, r2)
        if Xq is not None:
            Ko, Vo = oracle_read(run, st, c, Xq)
            ctx, layer = divmod(c, run.wl.n_layers)
            ek = record("swiglu", "K read", rel_fro(Kg[ctx, layer].float(), Ko), TOL)
            ev = record("swiglu", "V read", rel_fro(Vg[ctx, layer].float(), Vo), TOL)
            assert ek <= TOL and ev <= TOL, (c, ek, ev)


def test_swiglu_small_paper_mode_ragged_hidden_tiles():
    # 2 heads of 128, 96 hidden units (one hidden tile, 32 rows past F), 3 segments + a ragged tail
    wl = swiglu(n_ctx=2)
    run = DeviceRun(wl)
    run.ttl_context()
    check(run, range(wl.chains), wk.query_inputs(wl, "cuda"))
    run.close()


def test_swiglu_context_over_several_input_windows():
    # 64 segments a window: 3 full windows and a ragged fourth, each transformed after both
    # chain groups are done with the previous one
    wl = swiglu(n_ctx=1, N=3 * 64 * 128 + 70)
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    run.ttl_context()
    assert mone.mone_mem_kernel_time(run.h, mone.KERNEL_KINDS.index("prepass"))[1] == 4
    check(run, range(wl.chains), wk.query_inputs(wl, "cuda"))
    run.close()


def test_swiglu_read_with_silu_gate():
    # the read scales head h by SiLU(g_h) (the other reading of the gate), on the SwiGLU memory too
    wl = swiglu(n_ctx=1).replace(gate_act="silu")
    run = DeviceRun(wl)
    run.ttl_context()
    check(run, range(wl.chains), wk.query_inputs(wl, "cuda"))
    run.close()


def test_swiglu_paper_head_shape():
    # the paper's head shape: d = 896 as 4 heads of 224, 224 hidden units (k-blocks and hidden tiles
    # both run past 224), K || V = 2 x 7 heads of 64
    wl = swiglu(d=896, heads=4, F=224, n_kv=7, T=512, N=2 * 512 + 37, n_layers=3)
    run = DeviceRun(wl)
    run.ttl_context()
    check(run, range(wl.chains), wk.query_inputs(wl, "cuda"))
    run.close()


def test_swiglu_plain_mode():
    wl = swiglu(mode=wk.PLAIN, lr=0.05, N=2 * 128 + 17)
    run = DeviceRun(wl)
    run.ttl_context()
    check(run, range(wl.chains), wk.query_inputs(wl, "cuda"))
    run.close()


def test_swiglu_segment_with_caller_rates_and_loss():
    wl = swiglu(mode=wk.PLAIN, n_layers=3, lr=0.05, N=128)
    run = DeviceRun(wl)
    eta = wk.token_lr(wl, 1, 100, "cuda")
    loss = torch.zeros(1, device="cuda")
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, :100], run.K[0, 1, :100], run.V[0, 1, :100], 100, eta, loss)
    mone.mone_mem_sync(run.h)
    W1, W2, _, _ = run.state()
    X = O.f64(run.X[0, 1, :100])
    Y = np.concatenate([O.f64(run.K[0, 1, :100]), O.f64(run.V[0, 1, :100])], axis=1)
    st = oracle_init(wl, run.W1_0[1], run.W2_0[1])
    hp = O.Hyper(mode=wk.PLAIN, lr=wl.lr, memory="swiglu", n_heads=wl.heads)
    st, L = O.ttl_segment(st, X, Y, hp, None, eta=O.f64(eta))
    o1, o2 = gpu_layout(wl, st.W)
    assert rel_fro(W1[1], o1) <= TOL and rel_fro(W2[1], o2) <= TOL
    assert abs(loss.item() - L) <= TOL * max(1.0, abs(L))
    for c in (0, 2):  # untouched chains keep W_0 exactly
        assert torch.equal(W1[c], run.W1_0[c].cpu()) and torch.equal(W2[c], run.W2_0[c].cpu())
    run.close()


def test_swiglu_full_size_sampled_chains():
    # the paper's shape over its whole 32K-token context (64 segments), first and last layer
    wl = wk.WORKLOADS["swiglu_l24_d896_32k"]
    run = DeviceRun(wl)
    run.ttl_context()
    check(run, (0, 23), wk.query_inputs(wl, "cuda"))
    run.close()
    torch.cuda.empty_cache()
