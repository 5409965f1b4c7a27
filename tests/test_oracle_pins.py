"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these tests re-runs the oracle's own formula to check it: each one
uses an independent route (finite differences, a hand-derived closed form,
brute-force loops, an invariant), chosen so that a dropped term, a wrong sign,
a wrong index or a transposed operand in the oracle fails at least one.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rng(seed=0):
    return np.random.default_rng(seed)


def rand_mlp_state(r, d_in=8, d_hid=16, d_out=8):
    return O.init_state(W1=r.standard_normal((d_hid, d_in)) / math.sqrt(d_in),
                        W2=r.standard_normal((d_hid, d_out)) / math.sqrt(d_hid))


def rand_meta(r, d_in, n_heads=2, lr=1e-2, w_beta_scale=1.0):
    return O.Meta(alpha=1 + 0.1 * r.standard_normal(d_in), gamma=0.1 * r.standard_normal(d_in),
                  w_eta=0.5 * r.standard_normal(d_in) / math.sqrt(d_in), b_eta=math.log(math.expm1(lr)),
                  w_beta=w_beta_scale * r.standard_normal(d_in) / math.sqrt(d_in), b_beta=0.0,
                  gate=1 + 0.1 * r.standard_normal(n_heads))


# ----------------------------------------------------------------- scalar maps

def test_silu_prime_matches_finite_differences():
    z = np.linspace(-8, 8, 97)
    h = 1e-6
    fd = (O.silu(z + h) - O.silu(z - h)) / (2 * h)
    np.testing.assert_allclose(O.silu_prime(z), fd, rtol=0, atol=1e-9)


def test_scalar_special_values():
    assert O.sigmoid(0.0) == 0.5
    assert O.sigmoid(800.0) == 1.0 and O.sigmoid(-800.0) == 0.0
    assert abs(O.silu(math.log(3.0)) - 0.75 * math.log(3.0)) < 1e-15
    assert abs(O.softplus(math.log(math.expm1(0.01))) - 0.01) < 1e-15
    assert O.softplus(0.0) == math.log(2.0)


# ----------------------------------------------------------------- forward (Eq. 3) and loss (Eq. 7)

def test_mlp_forward_brute_force():
    r = rng(1)
    st = rand_mlp_state(r, 5, 7, 3)
    U = r.standard_normal((4, 5))
    out, _ = O.memory_forward(U, st.W, O.Hyper())
    W1, W2 = st.W["W1"], st.W["W2"]
    for j in range(4):
        for o in range(3):
            acc = 0.0
            for h in range(7):
                pre = sum(W1[h, i] * U[j, i] for i in range(5))
                acc += (pre / (1 + math.exp(-pre))) * W2[h, o]
            assert abs(out[j, o] - acc) < 1e-13


def test_swiglu_forward_brute_force():
    """Eq. 3: M(x) = W_out^T (SiLU(W_in x) * W_gate x), per head of width d_h."""
    r = rng(2)
    H, dh = 2, 3
    W = {"Win": r.standard_normal((H, dh, dh)), "Wg": r.standard_normal((H, dh, dh)),
         "Wout": r.standard_normal((H, dh, dh))}
    U = r.standard_normal((4, H * dh))
    out, _ = O.memory_forward(U, W, O.Hyper(memory="swiglu", n_heads=H))
    for j in range(4):
        for h in range(H):
            x = U[j, h * dh:(h + 1) * dh]
            z = []
            for a in range(dh):
                p = sum(W["Win"][h][a, i] * x[i] for i in range(dh))
                g = sum(W["Wg"][h][a, i] * x[i] for i in range(dh))
                z.append(p / (1 + math.exp(-p)) * g)
            for o in range(dh):
                ref = sum(W["Wout"][h][a, o] * z[a] for a in range(dh))
                assert abs(out[j, h * dh + o] - ref) < 1e-12


def test_onehot_closed_form_step():
    """Golden fixture derived by hand (tests/golden/make_onehot_fixture.py)."""
    with open(os.path.join(GOLDEN, "onehot_silu.json")) as f:
        fx = json.load(f)
    d, T, c = fx["d"], fx["T"], fx["c"]
    st = O.init_state(W1=c * np.eye(d), W2=np.eye(d))
    hp = O.Hyper(mode=O.PLAIN, lr=fx["eta"])
    assert abs(O.segment_loss(np.eye(d), np.eye(d), st.W, hp) - fx["loss"]) < 1e-15
    new, loss = O.ttl_segment(st, np.eye(d), np.eye(d), hp)
    assert abs(loss - fx["loss"]) < 1e-15
    off = ~np.eye(d, dtype=bool)
    np.testing.assert_allclose(np.diag(new.W["W1"]), fx["W1_diag_after"], rtol=0, atol=1e-15)
    np.testing.assert_allclose(np.diag(new.W["W2"]), fx["W2_diag_after"], rtol=0, atol=1e-15)
    assert np.all(new.W["W1"][off] == fx["offdiag_after"])
    assert np.all(new.W["W2"][off] == fx["offdiag_after"])


# ----------------------------------------------------------------- gradient (Eq. 10)

def _weighted_loss(U, Y, W, hp, eta):
    """F(W) = (1/T) sum_j eta_j l_j(W), from the forward only."""
    out, _ = O.memory_forward(U, W, hp)
    per = -np.sum(Y * out, axis=1) if hp.loss == "neg_inner" else 0.5 * np.sum((out - Y) ** 2, axis=1)
    return float(np.sum(eta * per) / U.shape[0])


@pytest.mark.parametrize("loss", ["neg_inner", "mse"])
def test_mlp_gradient_finite_differences(loss):
    r = rng(3)
    st = rand_mlp_state(r)
    U = r.standard_normal((4, 8))
    Y = r.standard_normal((4, 8))
    eta = 0.01 * (1 + r.random(4))
    hp = O.Hyper(loss=loss)
    G, _ = O.segment_gradient(U, Y, st.W, hp, eta)
    h = 1e-6
    for name in ("W1", "W2"):
        W = {k: v.copy() for k, v in st.W.items()}
        fd = np.zeros_like(W[name])
        for idx in np.ndindex(*W[name].shape):
            old = W[name][idx]
            W[name][idx] = old + h
            fp = _weighted_loss(U, Y, W, hp, eta)
            W[name][idx] = old - h
            fm = _weighted_loss(U, Y, W, hp, eta)
            W[name][idx] = old
            fd[idx] = (fp - fm) / (2 * h)
        err = np.linalg.norm(G[name] - fd) / np.linalg.norm(fd)
        assert err < 1e-7, (name, err)


def test_swiglu_gradient_finite_differences():
    r = rng(4)
    H, dh = 2, 3
    W = {"Win": r.standard_normal((H, dh, dh)), "Wg": r.standard_normal((H, dh, dh)),
         "Wout": r.standard_normal((H, dh, dh))}
    hp = O.Hyper(memory="swiglu", n_heads=H)
    U = r.standard_normal((5, H * dh))
    Y = r.standard_normal((5, H * dh))
    eta = np.full(5, 0.02)
    G, _ = O.segment_gradient(U, Y, W, hp, eta)
    h = 1e-6
    for name in W:
        fd = np.zeros_like(W[name])
        for idx in np.ndindex(*W[name].shape):
            old = W[name][idx]
            W[name][idx] = old + h
            fp = _weighted_loss(U, Y, W, hp, eta)
            W[name][idx] = old - h
            fm = _weighted_loss(U, Y, W, hp, eta)
            W[name][idx] = old
            fd[idx] = (fp - fm) / (2 * h)
        assert np.linalg.norm(G[name] - fd) / np.linalg.norm(fd) < 1e-7


def test_step_decreases_loss_to_first_order():
    """W_1 = W_0 - eta grad L gives L(W_1) - L(W_0) = -eta |grad L|^2 + O(eta^2)."""
    r = rng(5)
    st = rand_mlp_state(r)
    U = r.standard_normal((6, 8))
    Y = r.standard_normal((6, 8))
    for lr in (1e-4, 1e-5):
        hp = O.Hyper(mode=O.PLAIN, lr=lr)
        G, L0 = O.segment_gradient(U, Y, st.W, hp, np.full(6, lr))
        new, _ = O.ttl_segment(st, U, Y, hp)
        L1 = O.segment_loss(U, Y, new.W, hp)
        pred = -sum(np.sum(g * g) for g in G.values()) / lr
        assert L1 < L0
        assert abs((L1 - L0) / pred - 1) < 200 * lr


# ----------------------------------------------------------------- update (Eq. 8) closed forms

def test_linear_memory_hebbian_step():
    """Eq. 7 with M(u) = W u: grad l_j = -y_j u_j^T, so one step is
    W_1 = W_0 + (1/T) sum_j eta_j y_j u_j^T (a Hebbian outer-product write)."""
    r = rng(6)
    T, d_in, d_out = 5, 4, 3
    W0 = r.standard_normal((d_out, d_in))
    U = r.standard_normal((T, d_in))
    Y = r.standard_normal((T, d_out))
    eta = 0.01 * (1 + r.random(T))
    st = O.init_state(W=W0)
    new, _ = O.ttl_segment(st, U, Y, O.Hyper(mode=O.PLAIN, memory="linear"), eta=eta)
    ref = W0.copy()
    for j in range(T):
        for o in range(d_out):
            for i in range(d_in):
                ref[o, i] += eta[j] * Y[j, o] * U[j, i] / T
    np.testing.assert_allclose(new.W["W"], ref, rtol=0, atol=1e-15)


def test_linear_memory_delta_rule_step():
    """Squared-error loss on M(u) = W u: one step is the delta rule
    W_1 = W_0 - (1/T) sum_j eta_j (W_0 u_j - y_j) u_j^T."""
    r = rng(7)
    T, d_in, d_out = 6, 4, 5
    W0 = r.standard_normal((d_out, d_in))
    U = r.standard_normal((T, d_in))
    Y = r.standard_normal((T, d_out))
    eta = np.full(T, 0.05)
    st = O.init_state(W=W0)
    new, _ = O.ttl_segment(st, U, Y, O.Hyper(mode=O.PLAIN, memory="linear", loss="mse"), eta=eta)
    ref = W0.copy()
    for j in range(T):
        pred = [sum(W0[o, i] * U[j, i] for i in range(d_in)) for o in range(d_out)]
        for o in range(d_out):
            for i in range(d_in):
                ref[o, i] -= eta[j] * (pred[o] - Y[j, o]) * U[j, i] / T
    np.testing.assert_allclose(new.W["W"], ref, rtol=0, atol=1e-14)


def test_momentum_geometric_sum():
    """Constant gradient g and constant beta: mu_s = g (1 - beta^s)/(1 - beta),
    W_s = W_0 - g sum_{i<=s} (1 - beta^i)/(1 - beta).  A linear memory under
    Eq. 7 has a W-independent gradient, so replaying one segment gives constant g."""
    r = rng(8)
    T, d = 4, 6
    beta = 0.7
    meta = rand_meta(r, d, w_beta_scale=0.0)
    meta.b_beta = math.log(beta / (1 - beta))
    W0 = r.standard_normal((3, d))
    X = r.standard_normal((T, d))
    Y = r.standard_normal((T, 3))
    eta = np.full(T, 0.01)
    hp = O.Hyper(mode=O.PAPER, memory="linear", renorm=False)
    U = O.transform_inputs(X, hp, meta)
    g = np.zeros_like(W0)
    for j in range(T):
        g -= eta[j] * np.outer(Y[j], U[j]) / T
    st = O.init_state(W=W0)
    acc = 0.0
    for s in range(1, 8):
        st, _ = O.ttl_segment(st, X, Y, hp, meta, eta=eta)
        mu_ref = g * (1 - beta ** s) / (1 - beta)
        acc += (1 - beta ** s) / (1 - beta)
        np.testing.assert_allclose(st.mu["W"], mu_ref, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.W["W"], W0 - g * acc, rtol=1e-12, atol=1e-14)


def test_zero_learning_rate_leaves_weights_bit_identical():
    r = rng(9)
    st0 = rand_mlp_state(r, 8, 16, 8)
    X = r.standard_normal((12, 8))
    Y = r.standard_normal((12, 8))
    st, _ = O.ttl_context(st0.copy(), X, Y, 4, O.Hyper(mode=O.PLAIN, lr=0.0))
    for k in st.W:
        assert np.array_equal(st.W[k], st0.W[k])
    meta = rand_meta(r, 8, 4)
    st, _ = O.ttl_context(st0.copy(), X, Y, 4, O.Hyper(mode=O.PAPER), meta, eta=np.zeros(12))
    for k in st.W:
        assert np.array_equal(st.W[k], st0.W[k])
        assert not np.any(st.mu[k])


def test_renorm_keeps_initial_row_norms():
    r = rng(10)
    st = rand_mlp_state(r, 8, 16, 8)
    n1, n2 = O.row_norms(st.W["W1"]), O.row_norms(st.W["W2"])
    meta = rand_meta(r, 8, 4, lr=0.5)
    X = r.standard_normal((20, 8))
    Y = r.standard_normal((20, 8))
    st, _, trail = O.ttl_context(st, X, Y, 4, O.Hyper(mode=O.PAPER), meta, return_all=True)
    moved = 0.0
    for s in trail:
        np.testing.assert_allclose(O.row_norms(s.W["W1"]), n1, rtol=1e-13)
        np.testing.assert_allclose(O.row_norms(s.W["W2"]), n2, rtol=1e-13)
        moved = max(moved, np.abs(s.W["W1"] - trail[0].W["W1"]).max())
    assert moved > 1e-3


def _column_norms_by_loop(W):
    return np.array([math.sqrt(sum(W[h, c] ** 2 for h in range(W.shape[0]))) for c in range(W.shape[1])])


def test_output_channel_renorm_keeps_w1_rows_and_w2_columns():
    # R15: W1 keeps its row norms, W2 its column norms; W2's rows are free to move
    r = rng(21)
    st = rand_mlp_state(r, 8, 16, 8)
    n1, n2 = O.row_norms(st.W["W1"]), O.row_norms(st.W["W2"])
    c2 = _column_norms_by_loop(st.W["W2"])
    meta = rand_meta(r, 8, 4, lr=0.5)
    X = r.standard_normal((20, 8))
    Y = r.standard_normal((20, 8))
    _, _, trail = O.ttl_context(st, X, Y, 4, O.Hyper(mode=O.PAPER, renorm_axis="out"), meta, return_all=True)
    for s in trail:
        np.testing.assert_allclose(O.row_norms(s.W["W1"]), n1, rtol=1e-13)
        np.testing.assert_allclose(_column_norms_by_loop(s.W["W2"]), c2, rtol=1e-13)
    assert np.abs(O.row_norms(trail[-1].W["W2"]) - n2).max() > 1e-3


def test_output_channel_renorm_is_a_column_rescale_of_the_same_step():
    # one segment from the same state: W1, mu agree exactly with the row reading; each reading
    # rescales the same W2 - mu, by rows (ratios constant along a row) or by columns
    r = rng(22)
    st = rand_mlp_state(r, 8, 16, 8)
    meta = rand_meta(r, 8, 4, lr=0.5)
    X = r.standard_normal((4, 8))
    Y = r.standard_normal((4, 8))
    a, La = O.ttl_segment(st.copy(), X, Y, O.Hyper(mode=O.PAPER), meta)
    b, Lb = O.ttl_segment(st.copy(), X, Y, O.Hyper(mode=O.PAPER, renorm_axis="out"), meta)
    assert np.array_equal(a.W["W1"], b.W["W1"]) and np.array_equal(a.mu["W2"], b.mu["W2"]) and La == Lb
    raw = st.W["W2"] - a.mu["W2"]
    ra, rb = a.W["W2"] / raw, b.W["W2"] / raw
    np.testing.assert_allclose(ra, np.repeat(ra[:, :1], 8, axis=1), rtol=1e-12)
    np.testing.assert_allclose(rb, np.repeat(rb[:1, :], 16, axis=0), rtol=1e-12)
    assert np.abs(ra - rb).max() > 1e-3


def test_output_channel_renorm_zero_learning_rate_is_bit_identical():
    r = rng(23)
    st0 = rand_mlp_state(r, 8, 16, 8)
    X = r.standard_normal((12, 8))
    Y = r.standard_normal((12, 8))
    st, _ = O.ttl_context(st0.copy(), X, Y, 4, O.Hyper(mode=O.PAPER, renorm_axis="out"), rand_meta(r, 8, 4),
                          eta=np.zeros(12))
    for k in st.W:
        assert np.array_equal(st.W[k], st0.W[k])


# ----------------------------------------------------------------- prepass transforms (App. A)

def test_key_transform_unit_norm_and_plain_identity():
    r = rng(11)
    X = r.standard_normal((7, 8))
    meta = rand_meta(r, 8)
    U = O.transform_inputs(X, O.Hyper(mode=O.PAPER), meta)
    np.testing.assert_allclose(np.linalg.norm(U, axis=1), 1.0, rtol=1e-12)
    z = X * meta.alpha + meta.gamma
    z = z / (1 + np.exp(-z))
    cos = np.sum(U * z, axis=1) / np.linalg.norm(z, axis=1)
    np.testing.assert_allclose(cos, 1.0, rtol=1e-12)
    assert np.array_equal(O.transform_inputs(X, O.Hyper(mode=O.PLAIN), None), X)


def test_token_rate_and_decay_special_cases():
    r = rng(12)
    X = r.standard_normal((5, 8))
    meta = rand_meta(r, 8, lr=0.03)
    meta.w_eta[:] = 0
    np.testing.assert_allclose(O.token_rates(X, O.Hyper(mode=O.PAPER), meta), 0.03, rtol=1e-14)
    meta.w_beta[:] = 0
    assert O.momentum_decay(X, O.Hyper(mode=O.PAPER), meta) == 0.5
    assert O.momentum_decay(X, O.Hyper(mode=O.PLAIN), meta) == 0.0


def _rates_by_loop(X, meta):
    """eta_j = ln(1 + exp(sum_i w_i x_ji + b)) for every token j, by explicit loops."""
    out = []
    for j in range(X.shape[0]):
        z = meta.b_eta
        for i in range(X.shape[1]):
            z += meta.w_eta[i] * X[j, i]
        out.append(math.log1p(math.exp(z)))
    return np.array(out)


def _decay_by_loop(X, meta):
    """beta = 1 / (1 + exp(-(sum_i w_i (1/T') sum_j x_ji + b))), by explicit loops."""
    n, d = X.shape
    z = meta.b_beta
    for i in range(d):
        col = 0.0
        for j in range(n):
            col += X[j, i]
        z += meta.w_beta[i] * (col / n)
    return 1.0 / (1.0 + math.exp(-z))


def _transform_by_loop(X, meta):
    """u_j = z_j / sqrt(|z_j|^2 + 1e-12), z_ji = SiLU(alpha_i x_ji + gamma_i), by explicit loops."""
    U = np.empty_like(X)
    for j in range(X.shape[0]):
        z = []
        for i in range(X.shape[1]):
            a = meta.alpha[i] * X[j, i] + meta.gamma[i]
            z.append(a / (1.0 + math.exp(-a)))
        nrm = math.sqrt(sum(v * v for v in z) + 1e-12)
        for i in range(X.shape[1]):
            U[j, i] = z[i] / nrm
    return U


def _rate_inputs(seed):
    """Tokens with a clearly nonzero mean, so that a mean, a sum and a last token all differ,
    and meta-parameters whose data terms (w_eta . x, w_beta . mean x) are far from zero."""
    r = rng(seed)
    T, d = 6, 5
    X = 0.8 + r.standard_normal((T, d))
    meta = rand_meta(r, d, lr=0.05)
    meta.w_eta = 0.9 * r.standard_normal(d)
    meta.b_eta = 0.3
    meta.w_beta = 0.8 * r.standard_normal(d)
    meta.b_beta = -0.4
    return X, meta


def _pin_rates_and_decay():
    X, meta = _rate_inputs(40)
    hp = O.Hyper(mode=O.PAPER)
    rates = O.mone_oracle.token_rates(X, hp, meta)
    ref = _rates_by_loop(X, meta)
    assert rates.shape == ref.shape
    np.testing.assert_allclose(rates, ref, rtol=1e-13, atol=0)
    assert abs(O.mone_oracle.momentum_decay(X, hp, meta) - _decay_by_loop(X, meta)) < 1e-14


def _pin_two_segment_linear_memory():
    """Two paper-mode segments of a linear memory under Eq. 7, whose gradient does not
    depend on W: G_s = -(1/T) sum_j eta_sj y_sj u_sj^T, mu_1 = G_1, mu_2 = beta_2 mu_1 + G_2,
    W_s = W_{s-1} - mu_s (Eq. 8, App. A momentum).  Rates and decay come from the raw
    tokens x, the memory input from u = phi(x), each computed by loops."""
    X1, meta = _rate_inputs(41)
    r = rng(42)
    T, d = X1.shape
    X2 = -0.5 + 1.3 * r.standard_normal((T, d))
    Y1, Y2 = r.standard_normal((T, 3)), r.standard_normal((T, 3))
    W0 = r.standard_normal((3, d))
    hp = O.Hyper(mode=O.PAPER, memory="linear", renorm=False)
    st, _ = O.mone_oracle.ttl_context(O.init_state(W=W0), np.concatenate([X1, X2]), np.concatenate([Y1, Y2]), T,
                                      hp, meta)
    W, mu = W0.copy(), np.zeros_like(W0)
    for X, Y in ((X1, Y1), (X2, Y2)):
        U, eta, beta = _transform_by_loop(X, meta), _rates_by_loop(X, meta), _decay_by_loop(X, meta)
        G = np.zeros_like(W0)
        for j in range(T):
            for o in range(3):
                for i in range(d):
                    G[o, i] -= eta[j] * Y[j, o] * U[j, i] / T
        mu = beta * mu + G
        W = W - mu
    np.testing.assert_allclose(st.mu["W"], mu, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(st.W["W"], W, rtol=1e-12, atol=1e-15)


def test_token_rates_and_decay_by_loops():
    """Data-dependent terms of App. A's rate and decay (R3) element by element."""
    _pin_rates_and_decay()


def test_paper_mode_two_segments_of_a_linear_memory_by_loops():
    _pin_two_segment_linear_memory()


def _rates_from_u(X, hp, meta, eta=None):
    if eta is not None:
        return O.f64(eta)
    return O.softplus(O.transform_inputs(X, hp, meta) @ meta.w_eta + meta.b_eta)


def _rates_without_softplus(X, hp, meta, eta=None):
    if eta is not None:
        return O.f64(eta)
    return O.f64(X) @ meta.w_eta + meta.b_eta


def _decay_from_sum(X, hp, meta):
    return float(O.sigmoid(np.sum(O.f64(X), axis=0) @ meta.w_beta + meta.b_beta))


def _decay_from_last_token(X, hp, meta):
    return float(O.sigmoid(O.f64(X)[-1] @ meta.w_beta + meta.b_beta))


def _decay_from_u(X, hp, meta):
    return float(O.sigmoid(np.mean(O.transform_inputs(X, hp, meta), axis=0) @ meta.w_beta + meta.b_beta))


def _decay_wrong_axis(X, hp, meta):
    return float(O.sigmoid(np.mean(O.f64(X), axis=1) @ meta.w_beta[:X.shape[0]] + meta.b_beta))


@pytest.mark.parametrize("name,slip", [
    ("token_rates", _rates_from_u), ("token_rates", _rates_without_softplus),
    ("momentum_decay", _decay_from_sum), ("momentum_decay", _decay_from_last_token),
    ("momentum_decay", _decay_from_u), ("momentum_decay", _decay_wrong_axis)])
def test_planted_rate_and_decay_slips_fail_both_pins(monkeypatch, name, slip):
    """A plausible slip in the rate or the decay (the transformed u in place of x, a sum or
    the last token in place of the mean, the wrong pooling axis, a missing softplus),
    planted in the oracle, fails the direct pin and the two-segment pin."""
    monkeypatch.setattr(O.mone_oracle, name, slip)
    with pytest.raises((AssertionError, ValueError)):
        _pin_rates_and_decay()
    with pytest.raises((AssertionError, ValueError)):
        _pin_two_segment_linear_memory()


# ----------------------------------------------------------------- chain (Eq. 9)

def test_context_split_and_segment_loop_agree():
    r = rng(13)
    st0 = rand_mlp_state(r, 8, 16, 8)
    meta = rand_meta(r, 8, 4, lr=0.2)
    X = r.standard_normal((24, 8))
    Y = r.standard_normal((24, 8))
    hp = O.Hyper(mode=O.PAPER)
    full, _ = O.ttl_context(st0.copy(), X, Y, 4, hp, meta)
    a, _ = O.ttl_context(st0.copy(), X[:8], Y[:8], 4, hp, meta)
    b, _ = O.ttl_context(a, X[8:], Y[8:], 4, hp, meta)
    loop = st0.copy()
    for s in range(6):
        loop, _ = O.ttl_segment(loop, X[4 * s:4 * s + 4], Y[4 * s:4 * s + 4], hp, meta)
    for k in full.W:
        np.testing.assert_allclose(b.W[k], full.W[k], rtol=1e-13, atol=1e-15)
        np.testing.assert_allclose(loop.W[k], full.W[k], rtol=1e-13, atol=1e-15)


def test_partial_segment_averages_over_present_tokens():
    """Duplicating every token of a partial segment leaves a mean unchanged,
    so the step must be identical (it would differ under a fixed 1/T)."""
    r = rng(14)
    st0 = rand_mlp_state(r, 8, 16, 8)
    X = r.standard_normal((3, 8))
    Y = r.standard_normal((3, 8))
    hp = O.Hyper(mode=O.PLAIN, lr=0.1)
    a, la = O.ttl_segment(st0.copy(), X, Y, hp)
    b, lb = O.ttl_segment(st0.copy(), np.repeat(X, 2, axis=0), np.repeat(Y, 2, axis=0), hp)
    assert abs(la - lb) < 1e-14
    for k in a.W:
        np.testing.assert_allclose(a.W[k], b.W[k], rtol=1e-13, atol=1e-16)
    c, _, trail = O.ttl_context(st0.copy(), np.vstack([X, X, X[:1]]), np.vstack([Y, Y, Y[:1]]), 4, hp,
                                return_all=True)
    assert len(trail) == 2


# ----------------------------------------------------------------- read (Eq. 4 + normalisation)

def test_read_head_rms_equals_gate():
    r = rng(15)
    st = rand_mlp_state(r, 8, 16, 8)
    meta = rand_meta(r, 8, 4)
    Xq = r.standard_normal((5, 8))
    K, V = O.generate_kv(st, Xq, O.Hyper(mode=O.PAPER), meta, n_kv_heads=2, head_dim=2, eps=0.0)
    heads = np.concatenate([K, V])
    for h in range(4):
        rms = np.sqrt(np.mean(heads[h] ** 2, axis=1))
        np.testing.assert_allclose(rms, abs(meta.gate[h]), rtol=1e-13)


def test_read_silu_gate_rms_sign_and_zero_gate():
    # R16: each head's RMS is |SiLU(g_h)| (by hand: g / (1 + e^-g)), a zero gate silences the
    # head, and the output is the linear-gate output times SiLU(g) / g
    r = rng(24)
    st = rand_mlp_state(r, 8, 16, 8)
    meta = rand_meta(r, 8, 4)
    meta.gate = np.array([0.0, 1.0, -2.0, 3.0])
    Xq = r.standard_normal((5, 8))
    K, V = O.generate_kv(st, Xq, O.Hyper(mode=O.PAPER, gate_act="silu"), meta, n_kv_heads=2, head_dim=2, eps=0.0)
    Kl, Vl = O.generate_kv(st, Xq, O.Hyper(mode=O.PAPER), meta, n_kv_heads=2, head_dim=2, eps=0.0)
    heads, lin = np.concatenate([K, V]), np.concatenate([Kl, Vl])
    sg = [0.0, 1 / (1 + math.exp(-1.0)), -2 / (1 + math.exp(2.0)), 3 / (1 + math.exp(-3.0))]
    assert not np.any(heads[0])
    for h in range(1, 4):
        np.testing.assert_allclose(np.sqrt(np.mean(heads[h] ** 2, axis=1)), abs(sg[h]), rtol=1e-13)
        np.testing.assert_allclose(heads[h], lin[h] * (sg[h] / meta.gate[h]), rtol=1e-13)


def test_read_of_linear_memory_brute_force():
    """Linear memory, plain read: every head is a positive multiple of (W u)_head,
    the K half first, then the V half."""
    r = rng(16)
    W = r.standard_normal((8, 5))
    Xq = r.standard_normal((3, 5))
    K, V = O.generate_kv(O.init_state(W=W), Xq, O.Hyper(mode=O.PLAIN, memory="linear"), None, 2, 2, eps=0.0)
    heads = np.concatenate([K, V])
    for q in range(3):
        o = [sum(W[a, i] * Xq[q, i] for i in range(5)) for a in range(8)]
        for h in range(4):
            ref = np.array(o[2 * h:2 * h + 2])
            got = heads[h, q]
            assert abs(np.dot(ref, got) / (np.linalg.norm(ref) * np.linalg.norm(got)) - 1) < 1e-13
            assert abs(np.sqrt(np.mean(got ** 2)) - 1.0) < 1e-13


def test_swiglu_paper_mode_renorm_invariant():
    r = rng(17)
    H, dh = 2, 4
    W = {"Win": r.standard_normal((H, dh, dh)), "Wg": r.standard_normal((H, dh, dh)),
         "Wout": r.standard_normal((H, dh, dh))}
    st = O.init_state(**W)
    meta = rand_meta(r, H * dh, 2 * H, lr=0.3)
    X = r.standard_normal((8, H * dh))
    Y = r.standard_normal((8, H * dh))
    st, _ = O.ttl_context(st, X, Y, 4, O.Hyper(mode=O.PAPER, memory="swiglu", n_heads=H), meta)
    for k, w0 in W.items():
        for h in range(H):
            np.testing.assert_allclose(np.linalg.norm(st.W[k][h], axis=1), np.linalg.norm(w0[h], axis=1),
                                       rtol=1e-13)


# ----------------------------------------------------------------- consumer attention (Eq. 5, R14)

def _attn_inputs(n_q=4, n_kv=2, Lq=5, n_mem=3, dh=8, seed=0):
    r = np.random.default_rng(seed)
    return (r.standard_normal((n_q, Lq, dh)), r.standard_normal((n_kv, n_mem + Lq, dh)),
            r.standard_normal((n_kv, n_mem + Lq, dh)))


def test_attention_one_visible_key_returns_its_value():
    # no memory tokens: query token 0 sees only its own key, so its output is its own value
    Q, K, V = _attn_inputs(n_mem=0)
    out = O.attention(Q, K, V, 0)
    for h in range(Q.shape[0]):
        assert np.allclose(out[h, 0], V[h // 2, 0], rtol=0, atol=1e-14)


def test_attention_equal_keys_average_the_visible_values():
    Q, K, V = _attn_inputs()
    K[:] = K[:, :1]                      # every key identical -> uniform weights
    out = O.attention(Q, K, V, 3)
    for h in range(4):
        for i in range(5):
            assert np.allclose(out[h, i], V[h // 2, :3 + i + 1].mean(axis=0), atol=1e-12)


def test_attention_is_causal_over_query_tokens_and_sees_all_memory():
    Q, K, V = _attn_inputs()
    base = O.attention(Q, K, V, 3)
    K2, V2 = K.copy(), V.copy()
    K2[:, 3 + 4] += 5.0                  # the last query token's key and value
    V2[:, 3 + 4] -= 3.0
    out = O.attention(Q, K2, V2, 3)
    assert np.array_equal(out[:, :4], base[:, :4])          # earlier tokens do not see it
    assert not np.allclose(out[:, 4], base[:, 4])
    K3 = K.copy()
    K3[:, 0] += 5.0                      # a memory token changes every output
    out3 = O.attention(Q, K3, V, 3)
    assert all(not np.allclose(out3[:, i], base[:, i]) for i in range(5))


def test_attention_grouped_heads_and_softmax_by_hand():
    Q, K, V = _attn_inputs(n_q=6, n_kv=3, Lq=2, n_mem=2, dh=4, seed=3)
    out = O.attention(Q, K, V, 2)
    h, i = 3, 1                          # head 3 reads kv head 3 // 2 = 1 (not 3 % 3); token 1 sees 2 + 2 keys
    w = [np.exp(np.dot(Q[h, i], K[1, j]) / 2.0) for j in range(4)]
    want = sum(wj * V[1, j] for j, wj in enumerate(w)) / sum(w)
    assert np.allclose(out[h, i], want, atol=1e-13)
