"""Pure-Python brute force of one CLEAR-MoE FFN token (test infrastructure; tiny shapes only).

Per token and per output element, with Python floats and math.erf, in the factorised order
y_i = sum_k U[i][k] S[k] (sum_j Vh[k][j] z_j) + sum_j R_a[i][j] z_j: it never forms W_shared,
never sorts or permutes, and shares no code with `oracle.clearmoe`, so the two pin each other.
"""
from __future__ import annotations

import math


def _gelu(u: float) -> float:
    return u * 0.5 * (1.0 + math.erf(u / math.sqrt(2.0)))


def token_expert(x_t, Wg, bg) -> int:
    best_e, best = 0, None
    for e in range(len(Wg)):
        s = float(bg[e])
        for k in range(len(x_t)):
            s += float(Wg[e][k]) * float(x_t[k])
        if best is None or s > best:  # strict: an equal later logit never wins
            best_e, best = e, s
    return best_e


def mlp_token_expert(x_t, W_in, b_in, W_out, b_out, act: str) -> int:
    """Expert of one token under the MLP router W_out act(W_in x + b_in) + b_out."""
    h = []
    for j in range(len(W_in)):
        u = float(b_in[j])
        for k in range(len(x_t)):
            u += float(W_in[j][k]) * float(x_t[k])
        h.append(max(u, 0.0) if act == "relu" else _gelu(u))
    return token_expert(h, W_out, b_out)


def token_forward(x_t, W1, b1, U, S, Vh, residuals, e: int):
    H, d, r = len(W1), len(x_t), len(S)
    z = []
    for j in range(H):
        u = float(b1[j])
        for k in range(d):
            u += float(W1[j][k]) * float(x_t[k])
        z.append(_gelu(u))
    proj = []
    for k in range(r):
        s = 0.0
        for j in range(H):
            s += float(Vh[k][j]) * z[j]
        proj.append(float(S[k]) * s)
    R = residuals[e]
    y = []
    for i in range(len(U)):
        acc = 0.0
        for k in range(r):
            acc += float(U[i][k]) * proj[k]
        for j in range(H):
            acc += float(R[i][j]) * z[j]
        y.append(acc)
    return y


def dense_token(x_t, W1, b1, W2):
    """y_i = sum_j W2[i][j] GELU(W1 x_t + b1)_j: the unconverted layer on one token."""
    z = []
    for j in range(len(W1)):
        u = float(b1[j])
        for k in range(len(x_t)):
            u += float(W1[j][k]) * float(x_t[k])
        z.append(_gelu(u))
    return [sum(float(W2[i][j]) * z[j] for j in range(len(z))) for i in range(len(W2))]


def layer_ex(x, W1, b1, U, S, Vh, residuals, Wg, bg, W2, b2, cls_stride):
    """Tokens t with t % cls_stride == 0 (cls_stride > 0) take the dense layer and the group
    index len(residuals); the others as in `layer`; b2 (or None) is added to every output."""
    a, y = [], []
    for t, x_t in enumerate(x):
        if cls_stride > 0 and t % cls_stride == 0:
            e = len(residuals)
            row = dense_token(x_t, W1, b1, W2)
        else:
            e = token_expert(x_t, Wg, bg)
            row = token_forward(x_t, W1, b1, U, S, Vh, residuals, e)
        a.append(e)
        y.append([v + (float(b2[i]) if b2 is not None else 0.0) for i, v in enumerate(row)])
    return a, y


def layer(x, W1, b1, U, S, Vh, residuals, Wg, bg):
    """Returns (expert per token, output rows) for every token of x."""
    a, y = [], []
    for x_t in x:
        e = token_expert(x_t, Wg, bg)
        a.append(e)
        y.append(token_forward(x_t, W1, b1, U, S, Vh, residuals, e))
    return a, y
