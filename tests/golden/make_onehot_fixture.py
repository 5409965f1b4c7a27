"""Writes onehot_silu.json: a hand-derived closed-form TTL step (no oracle, no GPU).

Case: d_in = d_hid = d_out = 4, one segment of T = 4 tokens, plain mode with a
constant learning rate eta.  W1 = c I with c = ln 3 (so sigmoid(c) = 3/4
exactly), W2 = I, token j has u_j = e_j and target y_j = e_j.

By Eq. 3 (SiLU-MLP form) H = U W1^T = c I, A = SiLU(H) = (3c/4) I, O = A W2 = A.
Eq. 7: l_j = -y_j . o_j = -3c/4 for every j, so L_s = -3c/4.
Eq. 10 with per-token rate eta and the 1/T mean: dO = -(eta/T) Y.
  G2 = A^T dO = -(eta/T)(3c/4) I
  dA = dO W2^T = -(eta/T) I,  dH = dA * SiLU'(H);  SiLU'(c) = 3/4 (1 + c/4),
  off-diagonal dA = 0, so G1 = dH^T U = -(eta/T)(3/4)(1 + c/4) I.
Eq. 8 with beta = 0: W1_1 = W1 - G1, W2_1 = W2 - G2.
"""
import json
import math
import os

c = math.log(3.0)
eta, T = 0.01, 4
silu_c = 0.75 * c
dsilu_c = 0.75 * (1.0 + 0.25 * c)
fix = {
    "citation": "Eq. 3 (SiLU-MLP form), Eq. 7, Eq. 8, Eq. 10; plain-mode step",
    "d": 4, "T": T, "eta": eta, "c": c,
    "loss": -silu_c,
    "W1_diag_after": c + (eta / T) * dsilu_c,
    "W2_diag_after": 1.0 + (eta / T) * silu_c,
    "offdiag_after": 0.0,
}
with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "onehot_silu.json"), "w") as f:
    json.dump(fix, f, indent=1)
    f.write("\n")
