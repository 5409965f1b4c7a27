"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Tolerances: fp32 path, per-step relative Frobenius error of W1 and W2 <= 1e-4;
bf16 path, <= 2e-2 after the full context; the same bounds on the weight
*change* W_S - W_0, which is the part the kernels compute (and per hidden row:
1e-4 on the fp32 path, 8e-2 on the bf16 path); generated K/V <= 2e-2 (fp32
path: 1e-4).
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_17616_gb300 as mone
import workloads as wk
from harness import (DeviceRun, gpu_layout, oracle_chain, oracle_hyper, oracle_meta, oracle_read, record, rel_fro,
                     row_rel_errors)

pytestmark = pytest.mark.gpu

F32_TOL = 1e-4
BF16_TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_17616_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    mone.lib()


def small(mode, dtype="bf16", n_ctx=2, n_layers=2, d_in=256, d_hid=256, d_out=256, T=256, N=4 * 256 + 37, lr=0.3,
          hd=64, Q=40):
    return wk.Workload(f"small_{dtype}_{mode}", 10 + mode, n_ctx, n_layers, d_in, d_hid, d_out, d_out // (2 * hd), hd,
                       T, N, Q, dtype, mode, lr)


# The weight change W_S - W_0 is the part the kernels compute: it is held to the same bound as
# the weights (fp32: the per-step 1e-4; bf16: 2e-2 after the context), as a whole and, on the
# fp32 path, per hidden row.  On the bf16 path a row's change carries the bf16 rounding of its
# own operands only, so its error spreads wider than the whole matrix's (worst observed 3.9e-2
# against 4e-3); its bound, 8e-2, still fails a 128-row tile whose change is 10% off, which
# moves the whole-matrix figure by only about 3.5%.
DW_TOL = {F32_TOL: F32_TOL, BF16_TOL: BF16_TOL}
ROW_DW_TOL = {F32_TOL: F32_TOL, BF16_TOL: 8e-2}
# The momentum on the fp32 path: the same per-step bound as the weights.
MU_TOL = F32_TOL


def check_chain(run, chain, W1, W2, tol, n_tokens=None):
    st, _ = oracle_chain(run, chain, n_tokens)
    o1, o2 = gpu_layout(run.wl, st.W)
    name = "f32" if tol == F32_TOL else "bf16"
    e1 = record(name, "W1", rel_fro(W1[chain], o1), tol)
    e2 = record(name, "W2", rel_fro(W2[chain], o2), tol)
    w01, w02 = O.f64(run.W1_0[chain]), O.f64(run.W2_0[chain])
    g1, g2 = W1[chain].double().numpy() - w01, W2[chain].double().numpy() - w02
    d1 = record(name, "dW1", rel_fro(g1, o1 - w01), DW_TOL[tol])
    d2 = record(name, "dW2", rel_fro(g2, o2 - w02), DW_TOL[tol])
    r1 = record(name, "dW1 row", row_rel_errors(g1, o1 - w01).max(), ROW_DW_TOL[tol])
    r2 = record(name, "dW2 row", row_rel_errors(g2, o2 - w02).max(), ROW_DW_TOL[tol])
    assert e1 <= tol and e2 <= tol, (chain, e1, e2)
    assert d1 <= DW_TOL[tol] and d2 <= DW_TOL[tol], (chain, d1, d2)
    assert r1 <= ROW_DW_TOL[tol] and r2 <= ROW_DW_TOL[tol], (chain, r1, r2)
    return st


def check_mu(mu1, mu2, c, st, tol=MU_TOL):
    m1 = record("f32" if tol == MU_TOL else "bf16", "mu1", rel_fro(mu1[c], st.mu["W1"]), tol)
    m2 = record("f32" if tol == MU_TOL else "bf16", "mu2", rel_fro(mu2[c], st.mu["W2"]), tol)
    assert m1 <= tol and m2 <= tol, (c, m1, m2)


# ----------------------------------------------------------------- fp32 path (tiny workload)

def test_tiny_f32_per_step_parity_and_loss():
    wl = wk.WORKLOADS["tiny_f32"]
    run = DeviceRun(wl)
    _, losses, trail = oracle_chain(run, 0, return_all=True)
    loss_dev = torch.zeros(1, device="cuda")
    T = wl.seg_T
    for s in range(wl.S):
        sl = slice(s * T, (s + 1) * T)
        mone.mone_ttl_segment(run.h, 0, 0, run.X[0, 0, sl], run.K[0, 0, sl], run.V[0, 0, sl], T, None, loss_dev)
        mone.mone_mem_sync(run.h)
        W1, W2, _, _ = run.state()
        assert rel_fro(W1[0], trail[s].W["W1"]) <= F32_TOL, s
        assert rel_fro(W2[0], trail[s].W["W2"]) <= F32_TOL, s
        assert abs(loss_dev.item() - losses[s]) <= F32_TOL * max(1.0, abs(losses[s])), s
    run.close()


def test_tiny_f32_context_equals_segment_loop_and_read():
    wl = wk.WORKLOADS["tiny_f32"]
    a = DeviceRun(wl)
    a.ttl_context()
    W1a, W2a, _, _ = a.state()
    b = DeviceRun(wl)
    T = wl.seg_T
    for s in range(wl.S):
        sl = slice(s * T, (s + 1) * T)
        mone.mone_ttl_segment(b.h, 0, 0, b.X[0, 0, sl], b.K[0, 0, sl], b.V[0, 0, sl], T)
    mone.mone_mem_sync(b.h)
    W1b, W2b, _, _ = b.state()
    assert torch.equal(W1a, W1b) and torch.equal(W2a, W2b)
    st = check_chain(a, 0, W1a, W2a, F32_TOL)
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = a.generate_kv(Xq)
    Ko, Vo = oracle_read(a, st, 0, Xq)
    assert rel_fro(Kg[0, 0], Ko) <= F32_TOL and rel_fro(Vg[0, 0], Vo) <= F32_TOL
    a.close()
    b.close()


def test_f32_paper_mode_ragged():
    wl = small(wk.PAPER, "f32", T=128, N=3 * 128 + 50, d_in=128, d_hid=192, d_out=256, lr=0.5)
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, mu1, mu2 = run.state()
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, F32_TOL)
        check_mu(mu1, mu2, c, st)
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st, _ = oracle_chain(run, c)
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[c // 2, c % 2], Ko) <= F32_TOL and rel_fro(Vg[c // 2, c % 2], Vo) <= F32_TOL
    run.close()


def launches(run, kind):
    return mone.mone_mem_kernel_time(run.h, mone.KERNEL_KINDS.index(kind))[1]


def test_f32_mse_per_step_parity_and_loss():
    # the squared-error (delta-rule) variant on the fp32 path: per-step weights and loss at 1e-4
    wl = wk.WORKLOADS["tiny_f32"].replace(loss="mse", N=8 * 128)
    run = DeviceRun(wl)
    _, losses, trail = oracle_chain(run, 0, return_all=True)
    loss_dev = torch.zeros(1, device="cuda")
    T = wl.seg_T
    for s in range(wl.S):
        sl = slice(s * T, (s + 1) * T)
        mone.mone_ttl_segment(run.h, 0, 0, run.X[0, 0, sl], run.K[0, 0, sl], run.V[0, 0, sl], T, None, loss_dev)
        mone.mone_mem_sync(run.h)
        W1, W2, _, _ = run.state()
        assert rel_fro(W1[0], trail[s].W["W1"]) <= F32_TOL, s
        assert rel_fro(W2[0], trail[s].W["W2"]) <= F32_TOL, s
        assert abs(loss_dev.item() - losses[s]) <= F32_TOL * max(1.0, abs(losses[s])), s
    run.close()


def test_f32_mse_paper_ragged():
    wl = small(wk.PAPER, "f32", T=128, N=3 * 128 + 50, d_in=128, d_hid=192, d_out=256).replace(loss="mse")
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, mu1, mu2 = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, F32_TOL)
        check_mu(mu1, mu2, c, st)
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[c // 2, c % 2], Ko) <= F32_TOL and rel_fro(Vg[c // 2, c % 2], Vo) <= F32_TOL
    run.close()


def test_f32_tiled_path_paper_ragged():
    # d_in + d_out > 512: the rows stay in HBM and the per-segment fp32 phase kernels run
    wl = small(wk.PAPER, "f32", n_ctx=1, T=64, N=3 * 64 + 20, d_in=512, d_hid=128, d_out=256, lr=0.5)
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    run.ttl_context()
    assert launches(run, "resident") == 0 and launches(run, "phase_a") == wl.S
    W1, W2, mu1, mu2 = run.state()
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, F32_TOL)
        check_mu(mu1, mu2, c, st)
    run.close()


def test_f32_resident_segment_caller_rates_and_loss():
    # a partial segment of one chain with caller rates and the loss output, on the resident kernel
    wl = small(wk.PLAIN, "f32", n_ctx=1, n_layers=3, T=128, N=128)
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    eta = wk.token_lr(wl, 1, 100, "cuda")
    loss = torch.zeros(1, device="cuda")
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, :100], run.K[0, 1, :100], run.V[0, 1, :100], 100, eta, loss)
    mone.mone_mem_sync(run.h)
    assert launches(run, "resident") == 1 and launches(run, "phase_a") == 0
    W1, W2, _, _ = run.state()
    X = O.f64(run.X[0, 1, :100])
    Y = np.concatenate([O.f64(run.K[0, 1, :100]), O.f64(run.V[0, 1, :100])], axis=1)
    st = O.init_state(W1=O.f64(run.W1_0[1]), W2=O.f64(run.W2_0[1]))
    st, L = O.ttl_segment(st, X, Y, O.Hyper(mode=wk.PLAIN, lr=wl.lr), None, eta=O.f64(eta))
    assert rel_fro(W1[1], st.W["W1"]) <= F32_TOL and rel_fro(W2[1], st.W["W2"]) <= F32_TOL
    assert abs(loss.item() - L) <= F32_TOL * max(1.0, abs(L))
    for c in (0, 2):
        assert torch.equal(W1[c], run.W1_0[c].cpu()) and torch.equal(W2[c], run.W2_0[c].cpu())
    run.close()


def test_f32_resident_two_input_windows():
    # a paper-mode context longer than one input-transform window (64 segments): one resident
    # launch per window, the state handed from the first to the second through HBM
    wl = small(wk.PAPER, "f32", n_ctx=1, n_layers=2, T=64, N=64 * 64 + 64 + 40, d_in=64, d_hid=64, d_out=128,
               lr=0.5)
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    run.ttl_context()
    assert launches(run, "resident") == 2 and launches(run, "prepass") == 2
    W1, W2, mu1, mu2 = run.state()
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, F32_TOL)
        check_mu(mu1, mu2, c, st)
    run.close()


# ----------------------------------------------------------------- output-channel renorm, SiLU gate

@pytest.mark.parametrize("dtype,loss", [("bf16", "neg_inner"), ("bf16", "mse"), ("f32", "neg_inner"), ("f32", "mse")])
def test_output_channel_renorm_parity(dtype, loss):
    # W1 rows and W2 columns renormalised to their norms in W_0 (the other reading of App. A)
    if dtype == "bf16":
        wl = small(wk.PAPER, N=3 * 256 + 37).replace(renorm_axis="out", loss=loss)
    else:
        wl = small(wk.PAPER, "f32", T=128, N=3 * 128 + 50, d_in=128, d_hid=192, d_out=256,
                   lr=0.5).replace(renorm_axis="out", loss=loss)
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    run.ttl_context()
    assert launches(run, "resident") == 0
    W1, W2, _, _ = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, tol)
        col0 = run.W2_0[c].cpu().double().pow(2).sum(0).sqrt()
        row0 = run.W1_0[c].cpu().double().pow(2).sum(1).sqrt()
        assert torch.allclose(W2[c].double().pow(2).sum(0).sqrt(), col0, rtol=1e-5)
        assert torch.allclose(W1[c].double().pow(2).sum(1).sqrt(), row0, rtol=1e-5)
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[c // 2, c % 2].float(), Ko) <= tol and rel_fro(Vg[c // 2, c % 2].float(), Vo) <= tol
    run.close()


@pytest.mark.parametrize("dtype,mode", [("bf16", wk.PAPER), ("bf16", wk.PLAIN), ("f32", wk.PAPER)])
def test_silu_gate_read_parity(dtype, mode):
    # the read scales head h by SiLU(g_h); in plain mode without caller gates, by SiLU(1)
    if dtype == "bf16":
        wl = small(mode, N=2 * 256 + 10).replace(gate_act="silu")
    else:
        wl = small(mode, "f32", T=128, N=2 * 128 + 10, d_in=128, d_hid=192, d_out=256).replace(gate_act="silu")
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    run.ttl_context()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st, _ = oracle_chain(run, c)
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[c // 2, c % 2].float(), Ko) <= tol and rel_fro(Vg[c // 2, c % 2].float(), Vo) <= tol
    run.close()


# ----------------------------------------------------------------- contexts over several input windows

@pytest.mark.parametrize("dtype,loss", [("bf16", "neg_inner"), ("bf16", "mse"), ("f32", "neg_inner")])
def test_context_over_several_input_windows(dtype, loss):
    # paper mode transforms the input 64 segments at a time (one window), and both chain groups
    # join before each window's transform: 3 full windows and a ragged fourth (bf16, both losses),
    # and 2 + ragged on the fp32 tiled path
    if dtype == "bf16":
        wl = small(wk.PAPER, T=128, N=3 * 64 * 128 + 100).replace(loss=loss)
    else:
        wl = small(wk.PAPER, "f32", n_ctx=1, T=64, N=2 * 64 * 64 + 100, d_in=512, d_hid=128, d_out=256, lr=0.5)
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    mone.mone_mem_set_timing(run.h, 1)
    run.ttl_context()
    assert launches(run, "prepass") == -(-wl.S // 64)
    W1, W2, mu1, mu2 = run.state()
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, tol)
        if dtype == "f32":
            check_mu(mu1, mu2, c, st)
    run.close()


# ----------------------------------------------------------------- a zero learning rate

@pytest.mark.parametrize("dtype,shape", [("bf16", {}), ("f32", dict(d_in=128, d_hid=192, d_out=256, T=128)),
                                         ("f32", dict(d_in=512, d_hid=128, d_out=256, T=64))])
def test_zero_learning_rate_leaves_the_weights_bit_identical(dtype, shape):
    # plain mode with lr = 0: every gradient is exactly zero, so W comes back bit for bit (bf16
    # path, fp32 resident kernel, fp32 tiled kernels)
    wl = small(wk.PLAIN, dtype, lr=0.0, **shape)
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    assert torch.equal(W1, run.W1_0.cpu()) and torch.equal(W2, run.W2_0.cpu())
    run.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_zero_caller_rates_in_paper_mode_keep_the_state(dtype):
    # paper mode, caller rates all zero: the momentum stays exactly zero and W moves only by the
    # rounding of the renormalisation scale (n0 / |row|, both fp32 sums of the same row)
    n = 200 if dtype == "bf16" else 100  # one partial segment (T = 256 / 128)
    wl = _edge_small(dtype, n_ctx=1, T=256 if dtype == "bf16" else 128, N=n)
    run = DeviceRun(wl)
    eta = torch.zeros(n, device="cuda")
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, :n], run.K[0, 1, :n], run.V[0, 1, :n], n, eta)
    mone.mone_mem_sync(run.h)
    W1, W2, mu1, mu2 = run.state()
    assert not torch.any(mu1) and not torch.any(mu2)
    assert rel_fro(W1[1], O.f64(run.W1_0[1])) <= 1e-6 and rel_fro(W2[1], O.f64(run.W2_0[1])) <= 1e-6
    run.close()


# ----------------------------------------------------------------- edge sizes

def _edge_small(dtype, **kw):
    if dtype == "bf16":
        return small(wk.PAPER, **kw)
    return small(wk.PAPER, "f32", **{**dict(d_in=128, d_hid=192, d_out=256, lr=0.5), **kw})


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_context_shorter_than_a_segment_then_a_one_token_segment(dtype):
    wl = _edge_small(dtype, n_ctx=1, T=256 if dtype == "bf16" else 128, N=37)
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    run.ttl_context()                                        # one partial segment: T' = 37
    W1, W2, _, _ = run.state()
    for c in range(wl.chains):
        check_chain(run, c, W1, W2, tol)
    # then a segment of a single token (T' = 1) on chain 1
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, 36:37], run.K[0, 1, 36:37], run.V[0, 1, 36:37], 1)
    mone.mone_mem_sync(run.h)
    W1, W2, _, _ = run.state()
    st, _ = oracle_chain(run, 1)
    Y1 = np.concatenate([O.f64(run.K[0, 1, 36:37]), O.f64(run.V[0, 1, 36:37])], axis=1)
    st, _ = O.ttl_segment(st, O.f64(run.X[0, 1, 36:37]), Y1, oracle_hyper(wl), oracle_meta(run, 1))
    assert rel_fro(W1[1], st.W["W1"]) <= tol and rel_fro(W2[1], st.W["W2"]) <= tol
    run.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_largest_segment_T4096_ragged(dtype):
    # seg_T = 4096 (the largest the library takes) and a ragged second segment; on bf16 with
    # d_in = d_out = 256 phase B runs on CTA pairs, on fp32 the resident kernel streams 128 chunks
    wl = _edge_small(dtype, n_ctx=1, T=4096, N=4096 + 300)
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    for c in range(wl.chains):
        check_chain(run, c, W1, W2, tol)
    run.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_generate_kv_largest_query_4096(dtype):
    wl = _edge_small(dtype, n_ctx=1, n_layers=1, T=256 if dtype == "bf16" else 128, N=300, Q=4096)
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    run.ttl_context()
    Xq = wk.query_inputs(wl, "cuda")
    assert Xq.shape[2] == 4096
    Kg, Vg = run.generate_kv(Xq)
    st, _ = oracle_chain(run, 0)
    Ko, Vo = oracle_read(run, st, 0, Xq)
    assert rel_fro(Kg[0, 0].float(), Ko) <= tol and rel_fro(Vg[0, 0].float(), Vo) <= tol
    run.close()


# ----------------------------------------------------------------- bf16 tensor-core path (small shapes)

@pytest.mark.parametrize("mode", [wk.PLAIN, wk.PAPER])
def test_bf16_small_context_parity(mode):
    wl = small(mode)
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, mu1, mu2 = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, BF16_TOL)
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[c // 2, c % 2].float(), Ko) <= BF16_TOL
        assert rel_fro(Vg[c // 2, c % 2].float(), Vo) <= BF16_TOL
    run.close()


def test_bf16_segment_with_caller_rates_and_loss():
    wl = small(wk.PLAIN, n_ctx=1, n_layers=3, N=256)
    run = DeviceRun(wl)
    eta = wk.token_lr(wl, 1, 200, "cuda")
    loss = torch.zeros(1, device="cuda")
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, :200], run.K[0, 1, :200], run.V[0, 1, :200], 200, eta, loss)
    mone.mone_mem_sync(run.h)
    W1, W2, _, _ = run.state()
    X = O.f64(run.X[0, 1, :200])
    Y = np.concatenate([O.f64(run.K[0, 1, :200]), O.f64(run.V[0, 1, :200])], axis=1)
    st = O.init_state(W1=O.f64(run.W1_0[1]), W2=O.f64(run.W2_0[1]))
    st, L = O.ttl_segment(st, X, Y, O.Hyper(mode=wk.PLAIN, lr=wl.lr), None, eta=O.f64(eta))
    assert rel_fro(W1[1], st.W["W1"]) <= BF16_TOL and rel_fro(W2[1], st.W["W2"]) <= BF16_TOL
    assert record("bf16", "dW1 1 seg", rel_fro(W1[1].double() - run.W1_0[1].cpu().double(),
                                               st.W["W1"] - O.f64(run.W1_0[1])), 5e-2) <= 5e-2
    assert abs(loss.item() - L) <= BF16_TOL * max(1.0, abs(L))
    # untouched chains keep W_0 exactly
    for c in (0, 2):
        assert torch.equal(W1[c], run.W1_0[c].cpu()) and torch.equal(W2[c], run.W2_0[c].cpu())
    run.close()


def test_bf16_context_split_equals_whole():
    wl = small(wk.PAPER, N=6 * 256)
    a = DeviceRun(wl)
    a.ttl_context()
    b = DeviceRun(wl)
    n1 = 2 * 256
    X1, K1, V1 = (t[:, :, :n1].contiguous() for t in (b.X, b.K, b.V))
    X2, K2, V2 = (t[:, :, n1:].contiguous() for t in (b.X, b.K, b.V))
    b.ttl_context(X1, K1, V1, n1)
    b.ttl_context(X2, K2, V2, wl.N - n1)
    # equal up to bf16 operand rounding: the split run rounds the renormalised
    # weights at rest, the whole run rounds the raw weights and rescales in fp32
    for ta, tb in zip(a.state(), b.state()):
        assert rel_fro(tb, ta) <= 1e-3
    a.close()
    b.close()


def test_bf16_layer_permutation_permutes_results():
    wl = small(wk.PAPER, n_ctx=1, n_layers=4, N=512)
    a = DeviceRun(wl)
    a.ttl_context()
    W1a, W2a, _, _ = a.state()
    perm = [2, 0, 3, 1]
    b = DeviceRun(wl)
    mone.mone_mem_free(b.h)
    meta = {k: v[perm].contiguous() for k, v in a.meta.items()}
    from harness import config_of
    b.h = mone.mone_mem_init(config_of(wl), a.W1_0[perm].contiguous(), a.W2_0[perm].contiguous(), meta)
    b.ttl_context(a.X[:, perm].contiguous(), a.K[:, perm].contiguous(), a.V[:, perm].contiguous())
    W1b, W2b, _, _ = b.state()
    for i, p in enumerate(perm):
        assert rel_fro(W1b[i], W1a[p]) <= 1e-5 and rel_fro(W2b[i], W2a[p]) <= 1e-5
    a.close()
    b.close()


@pytest.mark.parametrize("mode", [wk.PLAIN, wk.PAPER])
def test_bf16_chain_groups_match_one_chain_handles(mode):
    """A call's chains run as two groups on two streams (here 2 + 1 chains; in paper
    mode three input-transform windows); every chain must match a handle that holds it alone."""
    # plain mode has no renormalisation and diverges over long contexts at this rate;
    # input-transform windows exist only in paper mode
    N = 2 * 64 * 128 + 300 if mode == wk.PAPER else 5 * 128 + 50
    wl = small(mode, n_ctx=1, n_layers=3, T=128, N=N)
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, mu1, mu2 = run.state()
    from harness import config_of
    one = wl.replace(n_layers=1)
    for c in range(wl.chains):
        meta = {k: v[c:c + 1].contiguous() for k, v in run.meta.items()} if run.meta else None
        h = mone.mone_mem_init(config_of(one), run.W1_0[c:c + 1].contiguous(), run.W2_0[c:c + 1].contiguous(), meta)
        X, K, V = (t[:, c:c + 1].contiguous() for t in (run.X, run.K, run.V))
        mone.mone_ttl_context(h, X, K, V, wl.N)
        st = [torch.empty_like(W1[c:c + 1], device="cuda"), torch.empty_like(W2[c:c + 1], device="cuda"),
              torch.empty_like(mu1[c:c + 1], device="cuda"), torch.empty_like(mu2[c:c + 1], device="cuda")]
        mone.mone_mem_read_state(h, *st)
        mone.mone_mem_sync(h)
        mone.mone_mem_free(h)
        # same arithmetic per chain; only the order of the row sum-of-squares atomics
        # differs, and its ulp-level effect on the renormalisation scale grows slowly
        # through the bf16 operand copy and the momentum over the 131 segments
        assert rel_fro(W1[c], st[0][0].cpu()) <= 2e-3 and rel_fro(W2[c], st[1][0].cpu()) <= 2e-3, c
        if mode == wk.PAPER:
            assert rel_fro(mu1[c], st[2][0].cpu()) <= 2e-2 and rel_fro(mu2[c], st[3][0].cpu()) <= 2e-2, c
        check_chain(run, c, W1, W2, BF16_TOL)
    run.close()


@pytest.mark.parametrize("Q,hd", [(200, 64), (131, 128)])
def test_bf16_generate_kv_several_query_tiles(Q, hd):
    """The tensor-core read takes queries 128 at a time: Q > 128 spans several tiles and a
    ragged last one (rows beyond Q are never written); hd = 128 puts one head per tile."""
    wl = small(wk.PAPER, n_ctx=1, n_layers=2, d_out=512, N=300, hd=hd, Q=Q)
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    assert Xq.shape[2] == Q
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st, _ = oracle_chain(run, c)
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[0, c].float(), Ko) <= BF16_TOL and rel_fro(Vg[0, c].float(), Vo) <= BF16_TOL
    run.close()


def test_generate_kv_into_strided_cache_and_reuse():
    wl = small(wk.PAPER, N=512)
    run = DeviceRun(wl)
    run.ttl_context()
    Q, off, S_tot = wl.Q, 7, wl.Q + 19
    Xq = wk.query_inputs(wl, "cuda")
    cache_k = torch.full((wl.n_ctx, wl.n_layers, wl.n_kv_heads, S_tot, wl.head_dim), 7.0, dtype=torch.bfloat16,
                         device="cuda")
    cache_v = cache_k.clone()
    strides = cache_k.stride()[:4]
    mone.mone_mem_generate_kv(run.h, Xq, Q, cache_k[:, :, :, off:], cache_v[:, :, :, off:], strides)
    mone.mone_mem_sync(run.h)
    Kd, Vd = run.generate_kv(Xq)
    assert torch.equal(cache_k[:, :, :, off:off + Q].cpu(), Kd) and torch.equal(cache_v[:, :, :, off:off + Q].cpu(), Vd)
    assert bool((cache_k[:, :, :, :off] == 7).all()) and bool((cache_k[:, :, :, off + Q:] == 7).all())
    K2, V2 = run.generate_kv(Xq)          # multi-query reuse: reading does not change the state
    assert torch.equal(K2, Kd) and torch.equal(V2, Vd)
    run.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_replayed_read_matches_the_launched_one_and_follows_the_state(dtype):
    # reads into the same buffers run as one captured graph from the second call on: the replay
    # equals the first (launched) read bit for bit, and after more learning it reads the new state
    wl = _edge_small(dtype, n_ctx=1, T=256 if dtype == "bf16" else 128, N=4 * (256 if dtype == "bf16" else 128) + 9)
    tol = F32_TOL if dtype == "f32" else BF16_TOL
    run = DeviceRun(wl)
    n1 = 2 * wl.seg_T
    X1, K1, V1 = (t[:, :, :n1].contiguous() for t in (run.X, run.K, run.V))
    X2, K2, V2 = (t[:, :, n1:].contiguous() for t in (run.X, run.K, run.V))
    run.ttl_context(X1, K1, V1, n1)
    Xq = wk.query_inputs(wl, "cuda")
    Ko = torch.empty(wl.n_ctx, wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim, dtype=Xq.dtype, device="cuda")
    Vo = torch.empty_like(Ko)
    strides = mone.kv_strides(wl.n_layers, wl.n_kv_heads, wl.Q, wl.head_dim)
    outs = []
    for _ in range(3):
        mone.mone_mem_generate_kv(run.h, Xq, wl.Q, Ko, Vo, strides)
        mone.mone_mem_sync(run.h)
        outs.append((Ko.clone(), Vo.clone()))
    for k, v in outs[1:]:
        assert torch.equal(k, outs[0][0]) and torch.equal(v, outs[0][1])
    run.ttl_context(X2, K2, V2, wl.N - n1)
    mone.mone_mem_generate_kv(run.h, Xq, wl.Q, Ko, Vo, strides)
    mone.mone_mem_sync(run.h)
    assert not torch.equal(Ko, outs[0][0])
    for c in range(wl.chains):
        st, _ = oracle_chain(run, c)
        Kr, Vr = oracle_read(run, st, c, Xq)
        assert rel_fro(Ko[0, c].float().cpu(), Kr) <= tol and rel_fro(Vo[0, c].float().cpu(), Vr) <= tol
    run.close()


# ----------------------------------------------------------------- CTA-pair phase B (segments of 1024 tokens and more)

@pytest.mark.parametrize("mode,loss,lr", [(wk.PLAIN, "neg_inner", 0.3), (wk.PAPER, "neg_inner", 0.3),
                                          (wk.PAPER, "mse", 0.3)])
def test_bf16_pair_phase_b_context_parity(mode, loss, lr):
    """From T = 1024 on, phase B runs on CTA pairs (256 columns x 256 hidden rows): 2 segments
    and a ragged tail, 3 chains in two groups (2 + 1)."""
    wl = small(mode, n_ctx=1, n_layers=3, T=1024, N=2 * 1024 + 300, lr=lr).replace(loss=loss)
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, mu1, mu2 = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, BF16_TOL)
        if mode == wk.PAPER:
            assert record("bf16", "mu1", rel_fro(mu1[c], st.mu["W1"]), 5e-2) <= 5e-2
            assert record("bf16", "mu2", rel_fro(mu2[c], st.mu["W2"]), 5e-2) <= 5e-2
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[0, c].float(), Ko) <= BF16_TOL and rel_fro(Vg[0, c].float(), Vo) <= BF16_TOL
    run.close()


def test_bf16_pair_phase_b_one_chain_segment():
    """A one-chain call (one group) through the pair kernel, with caller rates and the loss."""
    wl = small(wk.PLAIN, n_ctx=1, n_layers=2, T=1024, N=1024)
    run = DeviceRun(wl)
    eta = wk.token_lr(wl, 1, 900, "cuda")
    loss = torch.zeros(1, device="cuda")
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, :900], run.K[0, 1, :900], run.V[0, 1, :900], 900, eta, loss)
    mone.mone_mem_sync(run.h)
    W1, W2, _, _ = run.state()
    X = O.f64(run.X[0, 1, :900])
    Y = np.concatenate([O.f64(run.K[0, 1, :900]), O.f64(run.V[0, 1, :900])], axis=1)
    st = O.init_state(W1=O.f64(run.W1_0[1]), W2=O.f64(run.W2_0[1]))
    st, L = O.ttl_segment(st, X, Y, O.Hyper(mode=wk.PLAIN, lr=wl.lr), None, eta=O.f64(eta))
    assert rel_fro(W1[1], st.W["W1"]) <= BF16_TOL and rel_fro(W2[1], st.W["W2"]) <= BF16_TOL
    assert record("bf16", "dW1 1 seg", rel_fro(W1[1].double() - run.W1_0[1].cpu().double(),
                                               st.W["W1"] - O.f64(run.W1_0[1])), 5e-2) <= 5e-2
    assert abs(loss.item() - L) <= BF16_TOL * max(1.0, abs(L))
    assert torch.equal(W1[0], run.W1_0[0].cpu()) and torch.equal(W2[0], run.W2_0[0].cpu())
    run.close()


# ----------------------------------------------------------------- squared-error loss variant (bf16)

@pytest.mark.parametrize("mode,lr", [(wk.PLAIN, 0.01), (wk.PAPER, 0.3)])  # plain: the delta rule diverges at 0.05 for inputs of RMS 2
def test_bf16_mse_context_parity(mode, lr):
    """Loss 1/2 |M(u) - y|^2: the pre-pass forms y - M(u) at the segment's starting weights,
    then the same two phases run on it; 4 segments + a ragged tail, 4 chains in two groups."""
    wl = small(mode, lr=lr).replace(loss="mse")
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, mu1, mu2 = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in range(wl.chains):
        st = check_chain(run, c, W1, W2, BF16_TOL)
        if mode == wk.PAPER:
            assert record("bf16", "mu1", rel_fro(mu1[c], st.mu["W1"]), 5e-2) <= 5e-2
            assert record("bf16", "mu2", rel_fro(mu2[c], st.mu["W2"]), 5e-2) <= 5e-2
        Ko, Vo = oracle_read(run, st, c, Xq)
        assert rel_fro(Kg[c // 2, c % 2].float(), Ko) <= BF16_TOL
        assert rel_fro(Vg[c // 2, c % 2].float(), Vo) <= BF16_TOL
    run.close()


def test_bf16_mse_segment_with_caller_rates_and_loss():
    wl = small(wk.PLAIN, n_ctx=1, n_layers=3, N=256, lr=0.01).replace(loss="mse")
    run = DeviceRun(wl)
    eta = wk.token_lr(wl, 1, 200, "cuda")
    loss = torch.zeros(1, device="cuda")
    mone.mone_ttl_segment(run.h, 0, 1, run.X[0, 1, :200], run.K[0, 1, :200], run.V[0, 1, :200], 200, eta, loss)
    mone.mone_mem_sync(run.h)
    W1, W2, _, _ = run.state()
    X = O.f64(run.X[0, 1, :200])
    Y = np.concatenate([O.f64(run.K[0, 1, :200]), O.f64(run.V[0, 1, :200])], axis=1)
    st = O.init_state(W1=O.f64(run.W1_0[1]), W2=O.f64(run.W2_0[1]))
    st, L = O.ttl_segment(st, X, Y, O.Hyper(mode=wk.PLAIN, lr=wl.lr, loss="mse"), None, eta=O.f64(eta))
    assert rel_fro(W1[1], st.W["W1"]) <= BF16_TOL and rel_fro(W2[1], st.W["W2"]) <= BF16_TOL
    assert record("bf16", "dW1 1 seg", rel_fro(W1[1].double() - run.W1_0[1].cpu().double(),
                                               st.W["W1"] - O.f64(run.W1_0[1])), 5e-2) <= 5e-2
    assert abs(loss.item() - L) <= BF16_TOL * max(1.0, abs(L))
    for c in (0, 2):
        assert torch.equal(W1[c], run.W1_0[c].cpu()) and torch.equal(W2[c], run.W2_0[c].cpu())
    run.close()


def test_bf16_mse_chain_groups_match_one_chain_handles():
    wl = small(wk.PAPER, n_ctx=1, n_layers=3, T=128, N=2 * 64 * 128 + 300).replace(loss="mse")
    run = DeviceRun(wl)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    from harness import config_of
    one = wl.replace(n_layers=1)
    for c in range(wl.chains):
        meta = {k: v[c:c + 1].contiguous() for k, v in run.meta.items()}
        h = mone.mone_mem_init(config_of(one), run.W1_0[c:c + 1].contiguous(), run.W2_0[c:c + 1].contiguous(), meta)
        X, K, V = (t[:, c:c + 1].contiguous() for t in (run.X, run.K, run.V))
        mone.mone_ttl_context(h, X, K, V, wl.N)
        a1 = torch.empty_like(W1[c:c + 1], device="cuda")
        a2 = torch.empty_like(W2[c:c + 1], device="cuda")
        mone.mone_mem_read_state(h, a1, a2)
        mone.mone_mem_sync(h)
        mone.mone_mem_free(h)
        assert rel_fro(W1[c], a1[0].cpu()) <= 2e-3 and rel_fro(W2[c], a2[0].cpu()) <= 2e-3, c
        check_chain(run, c, W1, W2, BF16_TOL)
    run.close()


# ----------------------------------------------------------------- full-size workloads, sampled chains

# Every workload at its full context length (n_tokens None) in the launch configuration the
# bench times (all chains of the workload in one handle, two chain groups), the oracle
# replaying the sampled chains; the squared-error variant on a 16-segment prefix.
@pytest.mark.parametrize("name,chains,n_tokens,loss", [
    ("l16_d2048_128k", (0, 15), None, "neg_inner"),
    ("l16_d2048_128k", (9,), 8192, "mse"),
    ("l16_d2048_32k", (7,), None, "neg_inner"),
    ("l28_d3072_128k", (27,), None, "neg_inner"),
    ("ctx8_l16_T256", (77,), None, "neg_inner"),
    ("ctx8_l16_T512", (0, 127), None, "neg_inner"),
    ("ctx8_l16_T1024", (64,), None, "neg_inner"),
    ("ctx8_l16_T2048", (5,), None, "neg_inner"),
])
def test_full_size_sampled_chains(name, chains, n_tokens, loss):
    wl = wk.WORKLOADS[name].replace(loss=loss)
    run = DeviceRun(wl, n_tokens=n_tokens)
    run.ttl_context()
    W1, W2, _, _ = run.state()
    Xq = wk.query_inputs(wl, "cuda")
    Kg, Vg = run.generate_kv(Xq)
    for c in chains:
        st = check_chain(run, c, W1, W2, BF16_TOL)
        Ko, Vo = oracle_read(run, st, c, Xq)
        ctx, layer = divmod(c, wl.n_layers)
        assert rel_fro(Kg[ctx, layer].float(), Ko) <= BF16_TOL
        assert rel_fro(Vg[ctx, layer].float(), Vo) <= BF16_TOL
    run.close()
    torch.cuda.empty_cache()


# ----------------------------------------------------------------- per-segment metrics of a whole context

@pytest.mark.parametrize("case", ["bf16_paper", "bf16_mse", "f32_resident", "f32_tiled", "swiglu"])
def test_context_metrics_per_segment(case):
    # mone_ttl_context_metrics: per segment and chain, the loss L_s (Eq. 7, or the squared-error
    # variant) at the segment's starting weights and |mu_s|^2 (the Eq. 8 step), against the
    # oracle's per-segment losses and momenta; the state it leaves matches the oracle's
    if case == "bf16_paper":
        wl, tol = small(wk.PAPER), BF16_TOL
    elif case == "bf16_mse":
        wl, tol = small(wk.PAPER).replace(loss="mse"), BF16_TOL
    elif case == "f32_resident":
        wl, tol = wk.WORKLOADS["tiny_f32"].replace(N=8 * 128 + 50), F32_TOL
    elif case == "f32_tiled":
        wl, tol = small(wk.PAPER, "f32", n_ctx=1, T=64, N=3 * 64 + 20, d_in=512, d_hid=128, d_out=256, lr=0.5), F32_TOL
    else:
        wl, tol = wk.Workload("metrics_sw", 61, 1, 2, 256, 96, 256, 2, 64, 128, 3 * 128 + 50, 16, "bf16", wk.PAPER,
                              0.3, memory="swiglu", heads=2), BF16_TOL
    run = DeviceRun(wl)
    S = -(-wl.N // wl.seg_T)
    loss = torch.full((S, wl.chains), 7.0, device="cuda")
    step = torch.full((S, wl.chains), 7.0, device="cuda")
    mone.mone_ttl_context_metrics(run.h, run.X, run.K, run.V, wl.N, loss, step)
    mone.mone_mem_sync(run.h)
    W1, W2, _, _ = run.state()
    for c in range(wl.chains):
        check_chain(run, c, W1, W2, tol)
    loss, step = loss.cpu().double().numpy(), step.cpu().double().numpy()
    name = "f32" if tol == F32_TOL else "bf16"
    for c in range(wl.chains):
        _, losses, trail = oracle_chain(run, c, return_all=True)
        for s in range(S):
            L = losses[s]
            e = record(name, "seg loss", abs(loss[s, c] - L) / max(1.0, abs(L)), tol)
            assert e <= tol, (c, s, loss[s, c], L)
            m2 = sum(float(np.sum(v * v)) for v in trail[s].mu.values())
            e = record(name, "seg |mu|^2", abs(step[s, c] - m2) / m2, tol)
            assert e <= tol, (c, s, step[s, c], m2)
    run.close()
