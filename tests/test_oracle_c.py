"""The plain-C oracle (oracle/clearmoe_ref.c) against the paper's worked values and against the
other two restatements of the layer (CPU only).

The C oracle, the numpy oracle and the pure-Python brute force share no code. They must agree:
- the C oracle reproduces the hand-derived 3-token example (tests/golden/worked_example.json) and
  the GELU table, and its bf16 rounding is the numpy oracle's bit for bit;
- on random layers, every step (router logits, argmax with class tokens, the stable sort, fc1 +
  GELU, W_shared, the expert forward with class tokens and b2, the dense FFN, the MLP router, the
  LayerNorm) matches the numpy oracle to float64 rounding, the routing exactly;
- on tiny layers the C forward matches the brute force token by token.
"""
import json
import math
import pathlib

import numpy as np
import pytest

from oracle import brute as B
from oracle import clearmoe as O
from oracle import ref_c as C

GOLD = pathlib.Path(__file__).parent / "golden"


def _layer(rng, T, d, H, E, r):
    x = rng.standard_normal((T, d))
    W1 = rng.standard_normal((H, d)) / np.sqrt(d)
    b1 = 0.1 * rng.standard_normal(H)
    W2 = rng.standard_normal((d, H)) / np.sqrt(H)
    U, S, Vh = np.linalg.svd(W2, full_matrices=False)
    return dict(x=x, W1=W1, b1=b1, W2=W2, b2=0.1 * rng.standard_normal(d), U=U[:, :r], S=S[:r], Vh=Vh[:r],
                residuals=rng.standard_normal((E, d, H)) / np.sqrt(H), Wg=rng.standard_normal((E, d)),
                bg=rng.standard_normal(E))


def _rel(a, b):
    return np.linalg.norm(np.asarray(a) - np.asarray(b)) / max(np.linalg.norm(b), 1e-300)


def test_worked_example():
    g = json.loads((GOLD / "worked_example.json").read_text())
    env = dict(phi1=g["phi1"], phi2=g["phi2"])
    y_want = np.array([[float(eval(v, {}, env)) for v in row] for row in g["y"]])
    yd_want = np.array([[float(eval(v, {}, env)) for v in row] for row in g["y_dense"]])
    rt = C.route(g["x"], g["Wg"], g["bg"])
    assert rt["a"].tolist() == g["a"] and rt["counts"].tolist() == g["counts"]
    assert rt["offsets"].tolist() == g["offsets"] and rt["perm"].tolist() == g["perm"]
    y = C.ffn_forward(g["x"], g["W1"], g["b1"], g["U"], g["S"], g["Vh"], g["residuals"], rt["a"])
    assert np.max(np.abs(y - y_want)) <= 1e-15
    assert np.max(np.abs(C.dense_ffn(g["x"], g["W1"], g["b1"], g["W2"]) - yd_want)) <= 1e-15


def test_gelu_table_and_bf16_rounding():
    g = json.loads((GOLD / "gelu_normal_cdf.json").read_text())
    u = np.array([p[0] for p in g["points_u_phi"]])
    assert np.max(np.abs(C.gelu(u) - np.array([p[0] * p[1] for p in g["points_u_phi"]]))) <= 1e-15
    rng = np.random.default_rng(11)
    v = rng.standard_normal(20000) * np.exp(rng.uniform(-30, 30, 20000))
    halves = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 0.0, -0.0])
    for arr in (v, halves):
        assert np.array_equal(C.round_bf16(arr), O.to_bf16(arr))
    assert C.round_bf16(np.array([1.0 + 2.0 ** -8]))[0] == 1.0  # a half rounds to the even neighbour


@pytest.mark.parametrize("seed,T,d,H,E,r", [(0, 97, 24, 64, 4, 8), (1, 40, 16, 48, 3, 16), (2, 1, 8, 24, 2, 4)])
def test_steps_match_numpy_oracle(seed, T, d, H, E, r):
    L = _layer(np.random.default_rng(seed), T, d, H, E, r)
    lg = C.router_logits(L["x"], L["Wg"], L["bg"])
    assert _rel(lg, O.router_logits(L["x"], L["Wg"], L["bg"])) <= 1e-13
    a = C.argmax(lg)
    assert np.array_equal(a, O.argmax_lowest(O.router_logits(L["x"], L["Wg"], L["bg"])))
    srt, want = C.sort_by_group(a, E), O.sort_by_expert(a, E)
    for k in ("counts", "offsets", "perm"):
        assert np.array_equal(srt[k], want[k]), k
    z = C.fc1_gelu(L["x"], L["W1"], L["b1"])
    assert _rel(z, O.fc1_gelu(L["x"], L["W1"], L["b1"])) <= 1e-13
    assert np.array_equal(C.fc1_gelu(L["x"], L["W1"], L["b1"], True), O.to_bf16(z))  # z stored in bf16
    assert _rel(C.shared_weight(L["U"], L["S"], L["Vh"]), O.shared_weight(L["U"], L["S"], L["Vh"])) <= 1e-13
    y = C.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], a)
    assert _rel(y, O.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], a=a)) <= 1e-12
    yd = C.dense_ffn(L["x"], L["W1"], L["b1"], L["W2"], b2=L["b2"])
    assert _rel(yd, O.dense_ffn(L["x"], L["W1"], L["b1"], L["W2"], b2=L["b2"])) <= 1e-12
    assert _rel(C.layer_norm(L["x"]), O.layer_norm(L["x"])) <= 1e-13


def test_class_tokens_and_b2_match_numpy_oracle():
    L = _layer(np.random.default_rng(5), 60, 16, 40, 3, 8)
    cls = 7
    rt = C.route(L["x"], L["Wg"], L["bg"], cls)
    assert np.all(rt["a"][::cls] == 3) and rt["counts"][3] == math.ceil(60 / cls)
    assert np.array_equal(rt["perm"][60 - rt["counts"][3]:], np.arange(0, 60, cls))
    y = C.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], rt["a"],
                      W2=L["W2"], b2=L["b2"])
    want = O.ffn_forward_ex(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                            a=np.minimum(rt["a"], 2), W2=L["W2"], b2=L["b2"], cls_stride=cls)
    assert _rel(y, want) <= 1e-12


@pytest.mark.parametrize("act", ["relu", "gelu"])
def test_mlp_router_matches_numpy_oracle(act):
    rng = np.random.default_rng(9)
    x = rng.standard_normal((50, 24))
    W_in, b_in = rng.standard_normal((12, 24)) / 5, 0.1 * rng.standard_normal(12)
    W_out, b_out = rng.standard_normal((4, 12)), rng.standard_normal(4)
    lg = C.mlp_router_logits(x, W_in, b_in, W_out, b_out, act)
    assert _rel(lg, O.mlp_router_logits(x, W_in, b_in, W_out, b_out, act)) <= 1e-13
    assert np.array_equal(C.argmax(lg), [B.mlp_token_expert(x[t], W_in, b_in, W_out, b_out, act) for t in range(50)])


def test_forward_matches_brute_force():
    L = _layer(np.random.default_rng(3), 6, 5, 7, 3, 2)
    a = C.route(L["x"], L["Wg"], L["bg"])["a"]
    y = C.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], a)
    for t in range(6):
        assert a[t] == B.token_expert(L["x"][t], L["Wg"], L["bg"])
        want = B.token_forward(L["x"][t], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], int(a[t]))
        assert np.max(np.abs(y[t] - np.array(want))) <= 1e-13


def test_ties_bad_groups_and_empty_input():
    assert C.argmax(np.array([[1.0, 1.0, 0.5], [0.0, 2.0, 2.0]])).tolist() == [0, 1]  # lowest index wins
    with pytest.raises(ValueError):
        C.sort_by_group(np.array([0, 3]), 3)
    L = _layer(np.random.default_rng(4), 0, 8, 16, 2, 4)
    y = C.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], np.zeros(0, np.int64))
    assert y.shape == (0, 8)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_gpu_check_helper_on_the_numpy_oracle(dtype):
    """The GPU test's comparison against the C oracle, fed the numpy oracle's routing and output
    in place of the GPU's: it accepts them (to float64 rounding), and rejects a routing with one
    token moved to another expert and an output with one element off."""
    import synth
    from test_gpu_vs_c_oracle import check_against_c_oracle

    shape = synth.LayerShape(f"tiny_{dtype}", 160, 32, 128, 4, 8, dtype, n_cal=1500)
    L = synth.make_layer(shape)
    gr = O.route(L["x"], L["Wg"], L["bg"])
    y = O.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], a=gr["a"],
                      z_bf16=dtype == "bf16")
    assert check_against_c_oracle(L, y, gr) <= 1e-9
    assert check_against_c_oracle(L, y, gr, rows=np.arange(0, 160, 3)) <= 1e-9
    t = int(np.nonzero(~O.near_ties(L["x"], L["Wg"], L["bg"]))[0][0])
    moved = dict(gr, a=gr["a"].copy())
    moved["a"][t] = (moved["a"][t] + 1) % 4
    with pytest.raises(AssertionError):
        check_against_c_oracle(L, y, moved)
    y_bad = y.copy()
    y_bad[5, 3] += 1.0
    assert check_against_c_oracle(L, y_bad, gr) > 1e-2


def test_folded_and_scaled_forms_match_numpy_oracle():
    L = _layer(np.random.default_rng(8), 45, 16, 40, 3, 6)
    a = C.route(L["x"], L["Wg"], L["bg"])["a"]
    comb = C.fold_basis(L["U"], L["S"], L["Vh"], L["residuals"])
    assert _rel(comb, O.fold_basis(L["U"], L["S"], L["Vh"], L["residuals"])) <= 1e-13
    # the folded weights with a zero basis give the same layer as W_shared + residuals
    y_fold = C.ffn_forward(L["x"], L["W1"], L["b1"], np.zeros((16, 1)), np.zeros(1), np.zeros((1, 40)), comb, a)
    assert _rel(y_fold, C.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], a)) <= 1e-12
    R = L["W2"] - C.shared_weight(L["U"], L["S"], L["Vh"])
    s = np.array([0.5, 1.0, 2.0])
    y = C.ffn_forward_scaled(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], R, s, a)
    assert _rel(y, O.ffn_forward_scaled(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], R, s, a=a)) <= 1e-12
    # with every s_e = 1 the residuals are W2 - W_shared and the layer is the dense FFN
    y1 = C.ffn_forward_scaled(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], R, np.ones(3), a)
    assert _rel(y1, C.dense_ffn(L["x"], L["W1"], L["b1"], L["W2"])) <= 1e-12
    with pytest.raises(ValueError):
        C.ffn_forward_scaled(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], R, s, np.full(45, 3))
