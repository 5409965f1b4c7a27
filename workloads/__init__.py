"""Seeded synthetic workloads for the MoNe test-time-learning path.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic.  The oracle (``oracle/``) and the CUDA path both take
their inputs from here, so the two sides see identical values.

Shapes follow the five workload definitions of the build (tiny fp32 case,
16-layer 1B-class shape at 32K and 128K, 28-layer 3B-class shape at 128K, and
the 8-context batched sweep).  The paper evaluates on RULER (Sec. 4.1); no
dataset is used here: the activations stand in for a frozen backbone's
per-layer hidden states (Sec. 3.1) and the targets for its key/value
projections (Eq. 6), drawn as seeded random linear maps of the activations
plus 1% noise.

Seeds are counter-based: every tensor gets its own ``torch.Generator`` seeded
from (workload id, tensor kind, chain index), so any chain can be regenerated
alone, on any device, without drawing the others first.  Values drawn on CUDA
differ from values drawn on the CPU (different generators); tests that
compare the two paths draw once and copy.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch

PLAIN = 0
PAPER = 1


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload: layer/context counts, memory widths, segment plan."""

    name: str
    wid: int                 # workload id, mixed into every seed
    n_ctx: int
    n_layers: int
    d_in: int
    d_hid: int
    d_out: int               # = 2 * n_kv_heads * head_dim (K half then V half)
    n_kv_heads: int
    head_dim: int
    seg_T: int
    N: int                   # context tokens per chain
    Q: int                   # query tokens for generate_kv
    dtype: str               # "f32" or "bf16": activations and targets
    mode: int                # PLAIN or PAPER
    lr: float = 1e-2
    loss: str = "neg_inner"  # "neg_inner" (Eq. 7) or "mse" (squared-error variant)
    memory: str = "mlp"      # "mlp" (two-matrix SiLU MLP) or "swiglu" (per-head SwiGLU of Eq. 3)
    heads: int = 1           # swiglu heads: each sees d_in / heads input dimensions, d_hid hidden units
    renorm_axis: str = "rows"  # paper-mode renormalisation: "rows" of W1 and W2, or "out" (W1 rows, W2 columns)
    gate_act: str = "linear"   # read gate: g_h ("linear") or SiLU(g_h) ("silu")

    @property
    def chains(self) -> int:
        return self.n_ctx * self.n_layers

    @property
    def S(self) -> int:
        return -(-self.N // self.seg_T)

    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    def flops_per_token_per_layer(self) -> int:
        """Algorithmic work of one token on one chain: forward H, dA, dW1, dW2."""
        return 4 * (self.d_in * self.d_hid + self.d_hid * self.d_out)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    "tiny_f32": Workload("tiny_f32", 0, 1, 1, 256, 512, 256, 2, 64, 128, 4096, 32, "f32", PLAIN),
    "l16_d2048_32k": Workload("l16_d2048_32k", 1, 1, 16, 2048, 1024, 1024, 8, 64, 512, 32768, 64, "bf16", PAPER),
    "l16_d2048_128k": Workload("l16_d2048_128k", 2, 1, 16, 2048, 1024, 1024, 8, 64, 512, 131072, 64, "bf16", PAPER),
    "l28_d3072_128k": Workload("l28_d3072_128k", 3, 1, 28, 3072, 2048, 2048, 8, 128, 1024, 131072, 64, "bf16", PAPER),
}
# The paper's own memory (Eq. 3): per-head SwiGLU, d = 896 split into 4 heads of 224 with 224
# hidden units each, 24 layers; output [K || V] = 896 = 2 x 7 heads x 64.
WORKLOADS["swiglu_l24_d896_32k"] = Workload("swiglu_l24_d896_32k", 5, 1, 24, 896, 224, 896, 7, 64, 512, 32768, 64,
                                            "bf16", PAPER, memory="swiglu", heads=4)
for _T in (256, 512, 1024, 2048):
    WORKLOADS[f"ctx8_l16_T{_T}"] = Workload(f"ctx8_l16_T{_T}", 4, 8, 16, 2048, 1024, 1024, 8, 64, _T, 32768, 64,
                                            "bf16", PAPER)

_KIND = {"x": 1, "wt": 2, "noise": 3, "w1": 4, "w2": 5, "meta": 6, "q": 7, "eta": 8}


def _gen(wl: Workload, kind: str, chain: int, device) -> torch.Generator:
    seed = (wl.wid * 1_000_003 + _KIND[kind] * 10_007 + chain) & 0x7FFFFFFF
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def layer_rms(wl: Workload, chain: int) -> float:
    """Per-layer activation scale r_l = 0.5 + 1.5 l/(L-1); 1.0 for one-layer workloads."""
    if wl.n_layers == 1:
        return 1.0
    layer = chain % wl.n_layers
    return 0.5 + 1.5 * layer / (wl.n_layers - 1)


def chain_inputs(wl: Workload, chain: int, device="cpu", n_tokens: Optional[int] = None):
    """Activations X [n, d_in] and targets K, V [n, d_out/2] of one chain (context, layer).

    X ~ r_l N(0,1); Y = X W_t + 0.01 N(0,1) with W_t ~ N(0, 1/(r_l^2 d_in)) so
    that targets have unit RMS; K = Y[:, :d_out/2], V = Y[:, d_out/2:].  Values
    are rounded to the workload dtype once; Y is formed from the rounded X.
    """
    n = wl.N if n_tokens is None else n_tokens
    dt = wl.torch_dtype()
    r = layer_rms(wl, chain)
    x = torch.randn(n, wl.d_in, generator=_gen(wl, "x", chain, device), device=device) * r
    x = x.to(dt)
    wt = torch.randn(wl.d_in, wl.d_out, generator=_gen(wl, "wt", chain, device), device=device)
    wt = wt / (r * math.sqrt(wl.d_in))
    noise = torch.randn(n, wl.d_out, generator=_gen(wl, "noise", chain, device), device=device)
    y = torch.addmm(noise, x.float(), wt, beta=0.01).to(dt)
    half = wl.d_out // 2
    return x, y[:, :half].contiguous(), y[:, half:].contiguous()


def all_inputs(wl: Workload, device="cpu", n_tokens: Optional[int] = None):
    """X [n_ctx, n_layers, n, d_in], K, V [n_ctx, n_layers, n, d_out/2] for every chain."""
    n = wl.N if n_tokens is None else n_tokens
    dt = wl.torch_dtype()
    X = torch.empty(wl.n_ctx, wl.n_layers, n, wl.d_in, dtype=dt, device=device)
    K = torch.empty(wl.n_ctx, wl.n_layers, n, wl.d_out // 2, dtype=dt, device=device)
    V = torch.empty_like(K)
    for c in range(wl.chains):
        x, k, v = chain_inputs(wl, c, device, n)
        X[c // wl.n_layers, c % wl.n_layers] = x
        K[c // wl.n_layers, c % wl.n_layers] = k
        V[c // wl.n_layers, c % wl.n_layers] = v
    return X, K, V


def initial_weights(wl: Workload, device="cpu"):
    """W1_0 [chains, d_hid, d_in] ~ N(0, 1/d_in); W2_0 [chains, d_hid, d_out] ~ N(0, 1/d_hid); fp32.

    SwiGLU memory: W1_0 [chains, heads, 2 d_hid, dh] = [Win; Wg] per head ~ N(0, 1/dh) and
    W2_0 [chains, heads, d_hid, dh] = Wout ~ N(0, 1/d_hid), dh = d_in / heads."""
    if wl.memory == "swiglu":
        H, dh, F = wl.heads, wl.d_in // wl.heads, wl.d_hid
        W1 = torch.empty(wl.chains, H, 2 * F, dh, device=device)
        W2 = torch.empty(wl.chains, H, F, dh, device=device)
        for c in range(wl.chains):
            W1[c] = torch.randn(H, 2 * F, dh, generator=_gen(wl, "w1", c, device), device=device) / math.sqrt(dh)
            W2[c] = torch.randn(H, F, dh, generator=_gen(wl, "w2", c, device), device=device) / math.sqrt(F)
        return W1, W2
    W1 = torch.empty(wl.chains, wl.d_hid, wl.d_in, device=device)
    W2 = torch.empty(wl.chains, wl.d_hid, wl.d_out, device=device)
    for c in range(wl.chains):
        W1[c] = torch.randn(wl.d_hid, wl.d_in, generator=_gen(wl, "w1", c, device), device=device) / math.sqrt(wl.d_in)
        W2[c] = torch.randn(wl.d_hid, wl.d_out, generator=_gen(wl, "w2", c, device), device=device) / math.sqrt(wl.d_hid)
    return W1, W2


def meta_params(wl: Workload, device="cpu"):
    """Per-chain meta-parameters (fp32), standing in for the meta-trained ones (Sec. 3.3).

    alpha ~ 1 + 0.1 N(0,1), gamma ~ 0.1 N(0,1)          affine rescale of keys/queries
    w_eta ~ 0.5 N(0,1)/sqrt(d_in), b_eta = ln(e^lr - 1)  per-token learning rate (softplus)
    w_beta ~ N(0,1)/sqrt(d_in),    b_beta = 0            momentum decay (sigmoid)
    gate  ~ 1 + 0.1 N(0,1), one per output head (2 n_kv heads: K heads then V heads)
    """
    C, d = wl.chains, wl.d_in
    H = 2 * wl.n_kv_heads
    out = {k: torch.empty(C, d, device=device) for k in ("alpha", "gamma", "w_eta", "w_beta")}
    out["b_eta"] = torch.full((C,), math.log(math.expm1(wl.lr)), device=device)
    out["b_beta"] = torch.zeros(C, device=device)
    out["gate"] = torch.empty(C, H, device=device)
    for c in range(C):
        g = _gen(wl, "meta", c, device)
        out["alpha"][c] = 1.0 + 0.1 * torch.randn(d, generator=g, device=device)
        out["gamma"][c] = 0.1 * torch.randn(d, generator=g, device=device)
        out["w_eta"][c] = 0.5 * torch.randn(d, generator=g, device=device) / math.sqrt(d)
        out["w_beta"][c] = torch.randn(d, generator=g, device=device) / math.sqrt(d)
        out["gate"][c] = 1.0 + 0.1 * torch.randn(H, generator=g, device=device)
    return out


def query_inputs(wl: Workload, device="cpu", Q: Optional[int] = None):
    """Query hidden states Xq [n_ctx, n_layers, Q, d_in] ~ r_l N(0,1), workload dtype."""
    q = wl.Q if Q is None else Q
    Xq = torch.empty(wl.n_ctx, wl.n_layers, q, wl.d_in, dtype=wl.torch_dtype(), device=device)
    for c in range(wl.chains):
        x = torch.randn(q, wl.d_in, generator=_gen(wl, "q", c, device), device=device) * layer_rms(wl, c)
        Xq[c // wl.n_layers, c % wl.n_layers] = x.to(Xq.dtype)
    return Xq


def token_lr(wl: Workload, chain: int, n: int, device="cpu"):
    """A caller-supplied per-token learning rate, lr * U(0.5, 1.5), fp32 [n]."""
    g = _gen(wl, "eta", chain, device)
    return wl.lr * (0.5 + torch.rand(n, generator=g, device=device))
