"""fp64 CPU oracle of MoNe's test-time learning (TTL) and memory read.

TEST INFRASTRUCTURE ONLY.  Only tests, the smoke entry point and the CPU
baseline leg of the benchmark may import this module.  The product path (the
CUDA library and its binding) never calls it, and it shares no code with it.

Everything is plain NumPy in float64, written step by step in the order the
paper states the method, with library matmuls as the only building blocks.
Inputs may be float32 or bfloat16 values; they are upcast exactly.

Paper map (MoNe, "Modular Neural Memory for Efficient Long Context
Inference"):
  Sec. 3.1            segments of T tokens, s = 1..S, state W_0 -> W_S
  Eq. 3 (Sec. 3.2)    the memory network; the workloads use its two-matrix
                      SiLU-MLP form (rows of W1, W2 = hidden units, as Eq. 3
                      stores W_in / W_out); the three-matrix per-head SwiGLU of
                      Eq. 3 itself is implemented too (``memory="swiglu"``)
  Eq. 4               memory read h_j = M(phi(x_j); W_S)
  Sec. 3.2 (after Eq. 4), App. A
                      per-head RMSNorm of the read output, learned per-head gate
  Sec. 3.3, App. A    key/query transform: affine rescale -> SiLU -> L2 norm
  Eq. 7               loss l_{s,j} = -v^T M(k; W), segment mean L_s = (1/T) sum_j l
  Eq. 8               W_s = W_{s-1} - mu_s
  App. A              per-token learning rate (softplus), momentum decay
                      (sigmoid, from the chunk's hidden states), channel-wise
                      L2 renormalisation after each update
  Eq. 9-11            sequential chain over segments; gradient local to layer
  Eq. 2, Eq. 5        the consumer attention: softmax(q k^T / sqrt(d_h)) v over
                      [memory tokens || the query tokens' own keys]

Readings of passages the paper leaves open (each also listed in the design
notes):
  R1  M maps the hidden activations (width d_in) straight to [K || V]
      (width d_out); the backbone projections W_q, W_k, W_v are folded away.
  R2  Targets y_j = [k_j || v_j] are used as given (no SiLU/L2 on targets).
  R3  eta_j = softplus(w_eta . x_j + b_eta) scales token j's gradient;
      beta_s = sigmoid(w_beta . mean_j x_j + b_beta);
      mu_s = beta_s mu_{s-1} + sum_j (eta_j / T') grad l_j.
  R4  "Channel" = hidden unit = row of W1 and row of W2; each row is rescaled
      to its norm in W_0 after every update.
  R5  A last partial segment of T' < T tokens averages over T' tokens.
  R6  Read normalisation: each output head (width head_dim; K heads then V
      heads) is divided by sqrt(mean(o_h^2) + eps) and multiplied by a scalar
      gate g_h; eps = 1e-6.
  R7  Key/query transform u = z / sqrt(|z|^2 + 1e-12), z = SiLU(alpha*x + gamma).
  R8  Plain mode: u = x, eta_j = lr, beta = 0, no renormalisation.
  R13 The squared-error variant (loss="mse") replaces Eq. 7's l_j by
      1/2 |M(u_j) - y_j|^2 at the segment's starting weights; rates, momentum
      and renormalisation are unchanged.
  R14 Consumer attention (Eq. 5): the memory tokens are a prefix every query
      token sees; the query tokens are causal among themselves; query head h
      reads key/value head h // (n_q / n_kv) (grouped heads).
  R15 The other reading of "channel-wise" (App. A), renorm_axis="out": a channel is
      an output channel of each matrix, so W1 (hidden units out) keeps its rows and
      W2 (output features out) rescales each column to its norm in W_0.  MLP only.
  R16 The other reading of "SiLU-gated" (App. A), gate_act="silu": the learned
      per-head scalar gate enters the read through SiLU, o_h <- SiLU(g_h) o_h / rms.

Pinned by tests (tests/test_oracle_pins.py): the gradient (finite
differences), the loss (closed-form one-hot case), the update (closed form of
one step of a linear memory, Hebbian for Eq. 7 and the delta rule for a
squared-error loss), the momentum recurrence (geometric-sum closed form), the
renormalisation invariant (rows, and for R15 W1 rows and W2 columns), lr = 0
leaving W bit-identical, the read's RMS = |gate| invariant (R16: |SiLU(g)|, and
a zero output at g = 0), the read of a linear memory against brute force, and
the chain identities (context = loop of segments = split contexts), and the
consumer attention against its special cases (one visible key returns its
value, equal keys average the visible values, causality, grouped heads).
The data-dependent terms of R3 are pinned too: the rates and the decay against
explicit loops over tokens and features (nonzero w_eta, w_beta), and two
paper-mode segments of a linear memory against the same loops, so a rate taken
from u instead of x, or a decay pooled by a sum, the last token or the wrong
axis, fails.
Parity unpinned: the exact numbers of the paper-mode readings R3, R6, R7
(their forms are the build's reading; only the invariants above constrain
them).
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

PLAIN = 0
PAPER = 1

RMS_EPS = 1e-6      # R6
L2_EPS = 1e-12      # R7


# --------------------------------------------------------------------------- scalar maps

def sigmoid(z):
    """Logistic function, written through tanh so it cannot overflow."""
    z = np.asarray(z, dtype=np.float64)
    return 0.5 * (1.0 + np.tanh(0.5 * z))


def silu(z):
    """SiLU(z) = z * sigmoid(z) (Eq. 3)."""
    z = np.asarray(z, dtype=np.float64)
    return z * sigmoid(z)


def silu_prime(z):
    """d SiLU / dz = sigmoid(z) * (1 + z * (1 - sigmoid(z)))."""
    z = np.asarray(z, dtype=np.float64)
    s = sigmoid(z)
    return s * (1.0 + z * (1.0 - s))


def softplus(z):
    """softplus(z) = ln(1 + e^z) (App. A: per-token learning rate activation)."""
    return np.logaddexp(0.0, np.asarray(z, dtype=np.float64))


def f64(a):
    """Exact upcast of a float32 / bfloat16 array (NumPy or torch) to float64."""
    if hasattr(a, "detach"):
        a = a.detach().to("cpu").double().numpy()
    return np.array(a, dtype=np.float64)


# --------------------------------------------------------------------------- hyper-parameters and state

@dataclasses.dataclass
class Hyper:
    """How one chain learns.

    memory:  "mlp"    O = SiLU(U W1^T) W2                     (workload form of Eq. 3)
             "swiglu" per head: O_h = (SiLU(U_h Win^T) * (U_h Wg^T)) Wout   (Eq. 3)
             "linear" O = U W^T                              (closed-form checks only)
    loss:    "neg_inner" Eq. 7;  "mse" 0.5 |M(u) - y|^2 (delta-rule check only)
    """
    mode: int = PLAIN
    lr: float = 1e-2
    memory: str = "mlp"
    loss: str = "neg_inner"
    momentum: Optional[bool] = None     # default: on in PAPER mode
    renorm: Optional[bool] = None       # default: on in PAPER mode
    n_heads: int = 1                    # swiglu heads
    rms_eps: float = RMS_EPS
    renorm_axis: str = "rows"           # "rows" (R4) | "out": W1 rows, W2 columns (R15)
    gate_act: str = "linear"            # read gate g_h (R6) | "silu": SiLU(g_h) (R16)

    @property
    def use_momentum(self) -> bool:
        return (self.mode == PAPER) if self.momentum is None else self.momentum

    @property
    def use_renorm(self) -> bool:
        return (self.mode == PAPER) if self.renorm is None else self.renorm


@dataclasses.dataclass
class Meta:
    """Per-chain meta-parameters (App. A); all float64."""
    alpha: np.ndarray
    gamma: np.ndarray
    w_eta: np.ndarray
    b_eta: float
    w_beta: np.ndarray
    b_beta: float
    gate: np.ndarray

    @staticmethod
    def from_torch(m: dict, chain: int) -> "Meta":
        return Meta(f64(m["alpha"][chain]), f64(m["gamma"][chain]), f64(m["w_eta"][chain]),
                    float(m["b_eta"][chain]), f64(m["w_beta"][chain]), float(m["b_beta"][chain]),
                    f64(m["gate"][chain]))


@dataclasses.dataclass
class State:
    """Fast-weight state of one chain: weights, momentum, renorm targets (Sec. 3.3, App. A)."""
    W: dict            # name -> float64 array (rows = hidden units for mlp/swiglu)
    mu: dict
    n0: dict           # name -> row norms of W_0
    c0: dict = dataclasses.field(default_factory=dict)  # name -> column norms of W_0 (R15)

    def copy(self) -> "State":
        return State({k: v.copy() for k, v in self.W.items()},
                     {k: v.copy() for k, v in self.mu.items()},
                     {k: v.copy() for k, v in self.n0.items()},
                     {k: v.copy() for k, v in self.c0.items()})


def row_norms(W):
    return np.sqrt(np.sum(W * W, axis=-1))


def col_norms(W):
    return np.sqrt(np.sum(W * W, axis=-2))


def init_state(**W0) -> State:
    """W_0 given by the caller (learned in the paper, Sec. 3.3); mu_0 = 0."""
    W = {k: f64(v) for k, v in W0.items()}
    return State(W, {k: np.zeros_like(v) for k, v in W.items()}, {k: row_norms(v) for k, v in W.items()},
                 {k: col_norms(v) for k, v in W.items()})


# --------------------------------------------------------------------------- input transform (prepass)

def transform_inputs(X, hp: Hyper, meta: Optional[Meta]):
    """Memory input u_j (Sec. 3.3 / App. A; R7, R8)."""
    X = f64(X)
    if hp.mode == PLAIN:
        return X
    z = silu(meta.alpha * X + meta.gamma)
    return z / np.sqrt(np.sum(z * z, axis=1, keepdims=True) + L2_EPS)


def token_rates(X, hp: Hyper, meta: Optional[Meta], eta=None):
    """Per-token learning rate eta_j (App. A; R3, R8); a caller's eta wins."""
    X = f64(X)
    if eta is not None:
        return f64(eta)
    if hp.mode == PLAIN:
        return np.full(X.shape[0], hp.lr)
    return softplus(X @ meta.w_eta + meta.b_eta)


def momentum_decay(X, hp: Hyper, meta: Optional[Meta]) -> float:
    """beta_s in (0,1) from the chunk's hidden states (App. A; R3); 0 without momentum."""
    if not hp.use_momentum:
        return 0.0
    xbar = np.mean(f64(X), axis=0)
    return float(sigmoid(xbar @ meta.w_beta + meta.b_beta))


# --------------------------------------------------------------------------- memory network

def memory_forward(U, W: dict, hp: Hyper):
    """M(u; W) for every row of U, with the intermediates backprop needs."""
    if hp.memory == "mlp":
        Hh = U @ W["W1"].T
        A = silu(Hh)
        return A @ W["W2"], (Hh, A)
    if hp.memory == "linear":
        return U @ W["W"].T, None
    if hp.memory == "swiglu":
        n, d = U.shape
        dh = d // hp.n_heads
        O = np.empty((n, hp.n_heads * W["Wout"].shape[2]))
        cache = []
        for h in range(hp.n_heads):
            Uh = U[:, h * dh:(h + 1) * dh]
            P = Uh @ W["Win"][h].T          # W_in x
            Gt = Uh @ W["Wg"][h].T          # W_gate x
            Z = silu(P) * Gt
            O[:, h * dh:(h + 1) * dh] = Z @ W["Wout"][h]
            cache.append((Uh, P, Gt, Z))
        return O, cache
    raise ValueError(hp.memory)


def memory_backward(U, W: dict, hp: Hyper, cache, dO):
    """Gradient of sum_j dO_j . M(u_j; W) with respect to every fast weight (Eq. 10)."""
    if hp.memory == "mlp":
        Hh, A = cache
        G2 = A.T @ dO
        dA = dO @ W["W2"].T
        dH = dA * silu_prime(Hh)
        G1 = dH.T @ U
        return {"W1": G1, "W2": G2}
    if hp.memory == "linear":
        return {"W": dO.T @ U}
    if hp.memory == "swiglu":
        dh = U.shape[1] // hp.n_heads
        G = {k: np.zeros_like(v) for k, v in W.items()}
        for h, (Uh, P, Gt, Z) in enumerate(cache):
            dOh = dO[:, h * dh:(h + 1) * dh]
            G["Wout"][h] = Z.T @ dOh
            dZ = dOh @ W["Wout"][h].T
            dP = dZ * Gt * silu_prime(P)
            dG = dZ * silu(P)
            G["Win"][h] = dP.T @ Uh
            G["Wg"][h] = dG.T @ Uh
        return G
    raise ValueError(hp.memory)


def segment_loss(U, Y, W: dict, hp: Hyper) -> float:
    """L_s = (1/T') sum_j l_{s,j}; l = -y^T M(u) (Eq. 7) or 0.5|M(u) - y|^2 (mse check)."""
    O, _ = memory_forward(U, W, hp)
    if hp.loss == "neg_inner":
        per_tok = -np.sum(Y * O, axis=1)
    else:
        per_tok = 0.5 * np.sum((O - Y) ** 2, axis=1)
    return float(np.mean(per_tok))


def segment_gradient(U, Y, W: dict, hp: Hyper, eta):
    """sum_j (eta_j / T') grad_W l_{s,j}  (Eq. 10 with per-token rates, R3).

    Returns (gradient dict, loss L_s at W)."""
    n = U.shape[0]
    O, cache = memory_forward(U, W, hp)
    if hp.loss == "neg_inner":
        dL_dO = -Y                        # d l_j / d M(u_j) for Eq. 7
        per_tok = -np.sum(Y * O, axis=1)
    else:
        dL_dO = O - Y
        per_tok = 0.5 * np.sum((O - Y) ** 2, axis=1)
    dO = (eta / n)[:, None] * dL_dO
    return memory_backward(U, W, hp, cache, dO), float(np.mean(per_tok))


# --------------------------------------------------------------------------- one segment, one chain

def ttl_segment(state: State, X, Y, hp: Hyper, meta: Optional[Meta] = None, eta=None):
    """One TTL step W_{s-1} -> W_s on one segment (Eq. 7-8, App. A).  Returns (state, L_s)."""
    X = f64(X)
    Y = f64(Y)
    U = transform_inputs(X, hp, meta)
    rates = token_rates(X, hp, meta, eta)
    beta = momentum_decay(X, hp, meta)
    G, loss = segment_gradient(U, Y, state.W, hp, rates)
    new = state.copy()
    for k in new.W:
        new.mu[k] = beta * new.mu[k] + G[k]          # App. A momentum
        new.W[k] = new.W[k] - new.mu[k]              # Eq. 8
        if hp.use_renorm:                            # App. A, R4 (R15)
            Wk = new.W[k]
            if hp.renorm_axis == "out" and k == "W2":
                if hp.memory != "mlp":
                    raise ValueError("renorm_axis='out' is defined for the MLP memory")
                new.W[k] = Wk * (new.c0[k] / col_norms(Wk))[None, :]
            elif Wk.ndim == 2:
                new.W[k] = Wk * (new.n0[k] / row_norms(Wk))[:, None]
            else:
                for h in range(Wk.shape[0]):
                    Wk[h] = Wk[h] * (new.n0[k][h] / row_norms(Wk[h]))[:, None]
    return new, loss


def ttl_context(state: State, X, Y, T: int, hp: Hyper, meta: Optional[Meta] = None, eta=None,
                return_all: bool = False):
    """Chain W_0 -> W_1 -> ... -> W_S over consecutive segments of T tokens (Eq. 9).

    A last partial segment is allowed (R5).  With ``return_all`` the state after
    every segment is returned as well (for per-step parity)."""
    X = f64(X)
    Y = f64(Y)
    n = X.shape[0]
    trail, losses = [], []
    for s0 in range(0, n, T):
        s1 = min(n, s0 + T)
        e = None if eta is None else f64(eta)[s0:s1]
        state, loss = ttl_segment(state, X[s0:s1], Y[s0:s1], hp, meta, e)
        losses.append(loss)
        if return_all:
            trail.append(state.copy())
    return (state, losses, trail) if return_all else (state, losses)


# --------------------------------------------------------------------------- memory read

def generate_kv(state: State, Xq, hp: Hyper, meta: Optional[Meta], n_kv_heads: int, head_dim: int,
                eps: Optional[float] = None):
    """Memory tokens for a query (Eq. 4 and the normalisation after it; R6).

    Returns K_mem, V_mem each [n_kv_heads, Q, head_dim]."""
    eps = hp.rms_eps if eps is None else eps
    Uq = transform_inputs(Xq, hp, meta)
    O, _ = memory_forward(Uq, state.W, hp)
    Q = O.shape[0]
    n_heads = 2 * n_kv_heads
    out = np.empty((n_heads, Q, head_dim))
    gate = np.ones(n_heads) if meta is None else meta.gate
    if hp.gate_act == "silu":                        # R16
        gate = silu(gate)
    for h in range(n_heads):
        o = O[:, h * head_dim:(h + 1) * head_dim]
        rms = np.sqrt(np.mean(o * o, axis=1, keepdims=True) + eps)
        out[h] = gate[h] * o / rms
    return out[:n_kv_heads], out[n_kv_heads:]


# --------------------------------------------------------------------------- consumer attention

def attention(Q, K, V, n_mem: int):
    """Eq. 5 with Eq. 2 per head (R14): out[h, i] = softmax_j(q_{h,i} . k_j / sqrt(d_h)) v_j over the
    keys j visible to query token i: the n_mem memory tokens and query tokens 0..i.

    Q [n_q, Lq, d_h]; K, V [n_kv, n_mem + Lq, d_h] (memory tokens first); n_q a multiple of n_kv,
    query head h reading key/value head h // (n_q // n_kv).  Returns [n_q, Lq, d_h]."""
    Q, K, V = f64(Q), f64(K), f64(V)
    n_q, Lq, dh = Q.shape
    group = n_q // K.shape[0]
    out = np.empty((n_q, Lq, dh))
    for h in range(n_q):
        Kh, Vh = K[h // group], V[h // group]
        for i in range(Lq):
            vis = n_mem + i + 1                       # memory tokens, then query tokens up to i
            z = Kh[:vis] @ Q[h, i] / np.sqrt(dh)
            p = np.exp(z - z.max())
            out[h, i] = (p / p.sum()) @ Vh[:vis]
    return out

