"""Shared test plumbing: run a workload through the C ABI and through the oracle.

Inputs come from ``workloads`` (seeded); the GPU path is driven only through the
ctypes binding of libmone.so; the oracle is ``oracle`` (fp64 NumPy).  The two
never exchange intermediate values: both start from the same generated inputs.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle as O
import paper_2608_17616_gb300 as mone
import workloads as wk


def rel_fro(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


# Observed errors of every parity check of this session: (check, key, value, bound), printed
# at the end of the run (tests/conftest.py) so that the margins under each bound are visible.
MARGINS: list = []


def record(check: str, key: str, value: float, bound: float) -> float:
    MARGINS.append((check, key, float(value), float(bound)))
    return value


def row_rel_errors(a, b, floor=1e-6):
    """Per-row relative error |a_r - b_r| / |b_r| over the last axis (leading axes flattened);
    rows whose reference norm is below `floor` x the largest are skipped (nothing moved there)."""
    a = np.asarray(a, dtype=np.float64).reshape(-1, np.shape(a)[-1])
    b = np.asarray(b, dtype=np.float64).reshape(-1, np.shape(b)[-1])
    nb = np.linalg.norm(b, axis=1)
    keep = nb > floor * max(nb.max(), 1e-300)
    return np.linalg.norm(a - b, axis=1)[keep] / nb[keep]


def config_of(wl: wk.Workload) -> "mone.mone_config":
    return mone.make_config(wl.n_ctx, wl.n_layers, wl.d_in, wl.d_hid, wl.d_out, wl.n_kv_heads, wl.head_dim,
                            wl.seg_T, mone.MONE_FP32 if wl.dtype == "f32" else mone.MONE_BF16, wl.mode, wl.lr,
                            loss=mone.MONE_LOSS_MSE if wl.loss == "mse" else mone.MONE_LOSS_DOT,
                            memory=mone.MONE_MEM_SWIGLU if wl.memory == "swiglu" else mone.MONE_MEM_MLP,
                            mem_heads=wl.heads,
                            renorm_axis=mone.MONE_RENORM_OUT if wl.renorm_axis == "out" else mone.MONE_RENORM_ROWS,
                            gate_act=mone.MONE_GATE_SILU if wl.gate_act == "silu" else mone.MONE_GATE_LINEAR)


class DeviceRun:
    """A live libmone handle for one workload plus its generated device inputs."""

    def __init__(self, wl: wk.Workload, n_tokens=None, device="cuda"):
        self.wl = wl
        self.N = wl.N if n_tokens is None else n_tokens
        self.dev = device
        self.W1_0, self.W2_0 = wk.initial_weights(wl, device)
        self.meta = wk.meta_params(wl, device) if wl.mode == wk.PAPER else None
        self.X, self.K, self.V = wk.all_inputs(wl, device, self.N)
        self.h = mone.mone_mem_init(config_of(wl), self.W1_0, self.W2_0, self.meta)

    def close(self):
        if self.h:
            mone.mone_mem_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def state(self):
        W1 = torch.empty_like(self.W1_0)
        W2 = torch.empty_like(self.W2_0)
        mu1 = torch.empty_like(W1)
        mu2 = torch.empty_like(W2)
        mone.mone_mem_read_state(self.h, W1, W2, mu1, mu2)
        torch.cuda.synchronize()
        return W1.cpu(), W2.cpu(), mu1.cpu(), mu2.cpu()

    def ttl_context(self, X=None, K=None, V=None, N=None):
        X = self.X if X is None else X
        K = self.K if K is None else K
        V = self.V if V is None else V
        mone.mone_ttl_context(self.h, X, K, V, self.N if N is None else N)
        mone.mone_mem_sync(self.h)

    def generate_kv(self, Xq):
        wl = self.wl
        Q = Xq.shape[2]
        Kout = torch.empty(wl.n_ctx, wl.n_layers, wl.n_kv_heads, Q, wl.head_dim, dtype=Xq.dtype, device=self.dev)
        Vout = torch.empty_like(Kout)
        mone.mone_mem_generate_kv(self.h, Xq, Q, Kout, Vout, mone.kv_strides(wl.n_layers, wl.n_kv_heads, Q,
                                                                             wl.head_dim))
        mone.mone_mem_sync(self.h)
        return Kout.cpu(), Vout.cpu()


def oracle_hyper(wl: wk.Workload) -> O.Hyper:
    return O.Hyper(mode=wl.mode, lr=wl.lr, loss=wl.loss, memory=wl.memory, n_heads=wl.heads,
                   renorm_axis=wl.renorm_axis, gate_act=wl.gate_act)


def oracle_init(wl: wk.Workload, W1_0, W2_0) -> O.State:
    """Oracle state from one chain's W_0 in the library's layout."""
    if wl.memory == "swiglu":
        W1 = O.f64(W1_0)
        return O.init_state(Win=W1[:, :wl.d_hid], Wg=W1[:, wl.d_hid:], Wout=O.f64(W2_0))
    return O.init_state(W1=O.f64(W1_0), W2=O.f64(W2_0))


def gpu_layout(wl: wk.Workload, W: dict):
    """(W1, W2) of an oracle weight dict in the library's layout."""
    if wl.memory == "swiglu":
        return np.concatenate([W["Win"], W["Wg"]], axis=1), W["Wout"]
    return W["W1"], W["W2"]


def oracle_meta(run: DeviceRun, chain: int):
    return O.Meta.from_torch(run.meta, chain) if run.meta is not None else None


def oracle_chain(run: DeviceRun, chain: int, n_tokens=None, return_all=False):
    """Replay one chain in the oracle from the run's own generated inputs."""
    wl = run.wl
    n = run.N if n_tokens is None else n_tokens
    ctx, layer = divmod(chain, wl.n_layers)
    X = O.f64(run.X[ctx, layer, :n])
    Y = np.concatenate([O.f64(run.K[ctx, layer, :n]), O.f64(run.V[ctx, layer, :n])], axis=1)
    st = oracle_init(wl, run.W1_0[chain], run.W2_0[chain])
    return O.ttl_context(st, X, Y, wl.seg_T, oracle_hyper(wl), oracle_meta(run, chain), return_all=return_all)


def oracle_read(run: DeviceRun, state: O.State, chain: int, Xq):
    wl = run.wl
    ctx, layer = divmod(chain, wl.n_layers)
    return O.generate_kv(state, O.f64(Xq[ctx, layer]), oracle_hyper(wl), oracle_meta(run, chain),
                         wl.n_kv_heads, wl.head_dim)
