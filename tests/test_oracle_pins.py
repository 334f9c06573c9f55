"""Pins of the CPU oracle against facts fixed outside it (no GPU).

Each test checks the oracle against something other than itself: textbook values of the normal
CDF, a layer worked out by hand, the pure-Python brute force (factorised order, no sort), and
the algebraic identities the paper states (dense reduction, the D3 full-residual identity, the
scalar-residual form of Algorithm 2). The last test plants plausible mistakes in the oracle and
checks that some pin fails for each.
"""
import json
import pathlib

import numpy as np
import pytest

from oracle import brute as B
from oracle import clearmoe as O

GOLD = pathlib.Path(__file__).parent / "golden"


def _gold(name):
    return json.loads((GOLD / name).read_text())


def _eval(expr, env):
    return float(eval(expr, {}, env))  # golden expressions in phi1/phi2 only


def rel_err(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300)


def rand_layer(rng, T, d, H, E, r, res_scale=1.0):
    x = rng.standard_normal((T, d))
    W1 = rng.standard_normal((H, d)) / np.sqrt(d)
    b1 = 0.1 * rng.standard_normal(H)
    W2 = rng.standard_normal((d, H)) / np.sqrt(H)
    U, S, Vh = np.linalg.svd(W2, full_matrices=False)
    U, S, Vh = U[:, :r], S[:r], Vh[:r]
    res = res_scale * rng.standard_normal((E, d, H)) / np.sqrt(H)
    Wg = rng.standard_normal((E, d))
    bg = rng.standard_normal(E)
    return dict(x=x, W1=W1, b1=b1, W2=W2, U=U, S=S, Vh=Vh, residuals=res, Wg=Wg, bg=bg)


# ------------------------------------------------------------------ golden values
def check_gelu_table():
    g = _gold("gelu_normal_cdf.json")
    u = np.array([p[0] for p in g["points_u_phi"]])
    want = np.array([p[0] * p[1] for p in g["points_u_phi"]])
    return np.max(np.abs(O.gelu(u) - want)) <= 1e-15


def test_gelu_normal_cdf_table():
    assert check_gelu_table()


def check_worked_example():
    g = _gold("worked_example.json")
    env = dict(phi1=g["phi1"], phi2=g["phi2"])
    y_want = np.array([[_eval(v, env) for v in row] for row in g["y"]])
    yd_want = np.array([[_eval(v, env) for v in row] for row in g["y_dense"]])
    rt = O.route(g["x"], g["Wg"], g["bg"])
    ok = (rt["a"].tolist() == g["a"] and rt["counts"].tolist() == g["counts"]
          and rt["offsets"].tolist() == g["offsets"] and rt["perm"].tolist() == g["perm"])
    y = O.ffn_forward(g["x"], g["W1"], g["b1"], g["U"], g["S"], g["Vh"],
                      np.array(g["residuals"], float), g["Wg"], g["bg"])
    yd = O.dense_ffn(g["x"], g["W1"], g["b1"], g["W2"])
    return ok and np.max(np.abs(y - y_want)) <= 1e-15 and np.max(np.abs(yd - yd_want)) <= 1e-15


def test_worked_example():
    assert check_worked_example()


# ------------------------------------------------------------------ bf16 quantisation point
def test_to_bf16_matches_torch_and_ties():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    v = (rng.standard_normal(200000) * np.exp(rng.uniform(-20, 20, 200000))).astype(np.float32)
    want = torch.from_numpy(v).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.to_bf16(v.astype(np.float64)), want)
    # halfway cases round to the even neighbour
    assert O.to_bf16(1.0 + 2.0 ** -8) == 1.0
    assert O.to_bf16(1.0 + 3 * 2.0 ** -8) == 1.0 + 2.0 ** -6
    assert O.to_bf16(-(1.0 + 2.0 ** -8)) == -1.0


# ------------------------------------------------------------------ paper identities
def check_dense_reduction(seed=0):
    """E = 1, zero residual, full rank r = d: the layer is the dense FFN."""
    rng = np.random.default_rng(seed)
    d, H = 12, 40
    L = rand_layer(rng, 50, d, H, 1, d)
    y = O.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"],
                      np.zeros((1, d, H)), L["Wg"], L["bg"])
    return rel_err(y, O.dense_ffn(L["x"], L["W1"], L["b1"], L["W2"])) <= 1e-12


def test_dense_reduction():
    assert check_dense_reduction()


def check_d3_identity(seed=1):
    """Every residual = W2 - W_shared (D3): the dense FFN for any routing, random included."""
    rng = np.random.default_rng(seed)
    d, H, E, r = 10, 36, 3, 4
    L = rand_layer(rng, 64, d, H, E, r)
    D = L["W2"] - O.shared_weight(L["U"], L["S"], L["Vh"])
    a = rng.integers(0, E, 64)
    y = O.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], np.stack([D] * E), a=a)
    return rel_err(y, O.dense_ffn(L["x"], L["W1"], L["b1"], L["W2"])) <= 1e-12


def test_d3_identity_any_routing():
    assert check_d3_identity()


def check_scalar_residual(seed=2):
    """With W_e^res = (W2 - W_sh) s_e (Algorithm 2): y = (1 - s_a) W_sh z + s_a W2 z."""
    rng = np.random.default_rng(seed)
    d, H, E, r = 8, 32, 4, 3
    L = rand_layer(rng, 40, d, H, E, r)
    W_sh = O.shared_weight(L["U"], L["S"], L["Vh"])
    s = rng.uniform(0.5, 1.5, E)
    res = np.stack([(L["W2"] - W_sh) * s[e] for e in range(E)])
    y = O.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], res, L["Wg"], L["bg"])
    a = O.route(L["x"], L["Wg"], L["bg"])["a"]
    z = O.fc1_gelu(L["x"], L["W1"], L["b1"])
    want = (1 - s[a])[:, None] * (z @ W_sh.T) + s[a][:, None] * (z @ L["W2"].T)
    return rel_err(y, want) <= 1e-12


def test_scalar_residual_form():
    assert check_scalar_residual()


def check_fold_d3(seed=4):
    """Residuals W2 - W_shared (D3) fold to W2 itself for every expert."""
    rng = np.random.default_rng(seed)
    d, H, E, r = 9, 30, 3, 5
    L = rand_layer(rng, 8, d, H, E, r)
    D = L["W2"] - O.shared_weight(L["U"], L["S"], L["Vh"])
    W = O.fold_basis(L["U"], L["S"], L["Vh"], np.stack([D] * E))
    return all(np.max(np.abs(W[e] - L["W2"])) <= 1e-12 for e in range(E))


def check_folded_brute(seed=5, T=19, d=16, H=64, E=3, r=6):
    """The folded forward against the factorised brute force (which never forms W_shared)."""
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, T, d, H, E, r)
    a_b, y_b = B.layer(L["x"].tolist(), L["W1"].tolist(), L["b1"].tolist(), L["U"].tolist(),
                       L["S"].tolist(), L["Vh"].tolist(), L["residuals"].tolist(),
                       L["Wg"].tolist(), L["bg"].tolist())
    W = O.fold_basis(L["U"], L["S"], L["Vh"], L["residuals"])
    y = O.ffn_forward_folded(L["x"], L["W1"], L["b1"], W, a=np.array(a_b))
    return rel_err(y, np.array(y_b)) <= 1e-12


def test_fold_d3_gives_w2():
    assert check_fold_d3()


def test_folded_forward_brute_force():
    assert check_folded_brute()


# ------------------------------------------------------------------ fc2 bias and class tokens
def check_cls_all_dense(seed=6):
    """cls_stride = 1: every token is a class token, so the layer is the unconverted FFN (+ b2)
    whatever the residuals and the router say."""
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, 30, 12, 40, 3, 5)
    b2 = rng.standard_normal(12)
    y = O.ffn_forward_ex(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                         L["Wg"], L["bg"], W2=L["W2"], b2=b2, cls_stride=1)
    want = O.dense_ffn(L["x"], L["W1"], L["b1"], L["W2"]) + b2
    return rel_err(y, want) <= 1e-12


def check_cls_brute(seed=7, T=23, d=16, H=64, E=3, r=6, stride=5):
    """Class tokens and b2 against the pure-Python per-token loops (dense layer for t % 5 == 0)."""
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, T, d, H, E, r)
    b2 = rng.standard_normal(d)
    a_b, y_b = B.layer_ex(L["x"].tolist(), L["W1"].tolist(), L["b1"].tolist(), L["U"].tolist(),
                          L["S"].tolist(), L["Vh"].tolist(), L["residuals"].tolist(),
                          L["Wg"].tolist(), L["bg"].tolist(), L["W2"].tolist(), b2.tolist(), stride)
    rt = O.route_ex(L["x"], L["Wg"], L["bg"], stride)
    y = O.ffn_forward_ex(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                         a=np.array(a_b), W2=L["W2"], b2=b2, cls_stride=stride)
    free = ~rt["near_tie"]
    a_b = np.array(a_b)
    # slots: experts' tokens in (expert, id) order, then the class tokens in id order
    want_perm = np.array(sorted(range(T), key=lambda t: (a_b[t], t)))
    return (np.array_equal(rt["a"][free], a_b[free]) and np.array_equal(rt["perm"], want_perm)
            and rt["counts"][E] == len(range(0, T, stride)) and rel_err(y, np.array(y_b)) <= 1e-12)


def check_cls_keeps_routed_rows(seed=8):
    """Rows of routed tokens are those of Eq. 2 (ffn_forward) shifted by b2; class rows differ."""
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, 40, 10, 36, 4, 4)
    b2 = rng.standard_normal(10)
    args = (L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], L["Wg"], L["bg"])
    y0 = O.ffn_forward(*args)
    y = O.ffn_forward_ex(*args, W2=L["W2"], b2=b2, cls_stride=7)
    cls = np.arange(40) % 7 == 0
    return (np.max(np.abs(y[~cls] - b2 - y0[~cls])) <= 1e-12
            and np.min(np.abs(y[cls] - b2 - y0[cls]).max(axis=1)) > 1e-6)


def test_class_tokens_all_dense():
    assert check_cls_all_dense()


def test_class_tokens_and_b2_brute_force():
    assert check_cls_brute()
    assert check_cls_brute(seed=9, T=9, stride=1)   # all class tokens
    assert check_cls_brute(seed=10, T=5, stride=8)  # one class token, T < stride


def test_class_tokens_keep_routed_rows():
    assert check_cls_keeps_routed_rows()


def test_routing_with_class_tokens_invariants():
    rng = np.random.default_rng(11)
    L = rand_layer(rng, 197 * 3, 8, 16, 5, 2)
    rt = O.route_ex(L["x"], L["Wg"], L["bg"], 197)
    T = 197 * 3
    assert np.array_equal(rt["a"][[0, 197, 394]], [5, 5, 5]) and rt["counts"][5] == 3
    assert rt["offsets"][5] == T - 3 and rt["offsets"][6] == T
    assert np.array_equal(rt["perm"][T - 3:], [0, 197, 394])
    assert np.array_equal(np.sort(rt["perm"]), np.arange(T))


# ------------------------------------------------------------------ MLP router
def check_mlp_identity(seed=12):
    """W_in = [I; -I], b_in = 0, W_out = [W_g, -W_g], b_out = b_g: since act(u) - act(-u) = u for
    ReLU and for GELU, the MLP router's logits are the linear router's."""
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, 40, 9, 20, 5, 3)
    d = 9
    W_in = np.concatenate([np.eye(d), -np.eye(d)])
    W_out = np.concatenate([L["Wg"], -L["Wg"]], axis=1)
    want = O.router_logits(L["x"], L["Wg"], L["bg"])
    return all(rel_err(O.mlp_router_logits(L["x"], W_in, np.zeros(2 * d), W_out, L["bg"], act), want)
               <= 1e-12 for act in ("relu", "gelu"))


def check_mlp_brute(seed=13, T=40, d=12, hidden=6, E=4):
    """route_mlp against the pure-Python per-token loops, both activations."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, d))
    W_in, b_in = rng.standard_normal((hidden, d)), rng.standard_normal(hidden)
    W_out, b_out = rng.standard_normal((E, hidden)), rng.standard_normal(E)
    ok = True
    for act in ("relu", "gelu"):
        rt = O.route_mlp(x, W_in, b_in, W_out, b_out, act)
        a_b = np.array([B.mlp_token_expert(x[t].tolist(), W_in.tolist(), b_in.tolist(), W_out.tolist(),
                                           b_out.tolist(), act) for t in range(T)])
        free = ~rt["near_tie"]
        ok = ok and np.array_equal(rt["a"][free], a_b[free]) and free.sum() >= T - 2
    return ok


def test_mlp_router_reduces_to_linear():
    assert check_mlp_identity()


def test_mlp_router_brute_force():
    assert check_mlp_brute()
    assert check_mlp_brute(seed=14, T=64, d=16, hidden=16, E=7)


def test_mlp_router_generator_routes_like_linear():
    import synth
    L = synth.make_layer(synth.DEIT_TINY_FP32.with_(T=600, n_cal=2000))
    M = synth.mlp_router(L)
    a_lin = O.route(L["x"], L["Wg"], L["bg"])["a"]
    a_mlp = O.route_mlp(L["x"], M["W_in"], M["b_in"], M["W_out"], M["b_out"])["a"]
    assert M["hidden"] == 32 and np.mean(a_lin == a_mlp) > 0.9


# ------------------------------------------------------------------ scalar residuals (Algorithm 2)
def check_scaled_brute(seed=15, T=21, d=12, H=48, E=3, r=5):
    """W_e^res = s_e R: the one-matrix form against the brute force on the E scaled copies."""
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, T, d, H, E, r)
    R = rng.standard_normal((d, H)) / np.sqrt(H)
    s = rng.uniform(0.3, 1.7, E)
    res = [s[e] * R for e in range(E)]
    a_b, y_b = B.layer(L["x"].tolist(), L["W1"].tolist(), L["b1"].tolist(), L["U"].tolist(),
                       L["S"].tolist(), L["Vh"].tolist(), [m.tolist() for m in res],
                       L["Wg"].tolist(), L["bg"].tolist())
    y = O.ffn_forward_scaled(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], R, s, a=np.array(a_b))
    return rel_err(y, np.array(y_b)) <= 1e-12


def test_scaled_residual_form_brute_force():
    assert check_scaled_brute()
    assert check_scaled_brute(seed=16, T=8, E=1)


# ------------------------------------------------------------------ brute force
def check_brute(seed, T=23, d=16, H=64, E=4, r=16):
    rng = np.random.default_rng(seed)
    L = rand_layer(rng, T, d, H, E, r)
    a_b, y_b = B.layer(L["x"].tolist(), L["W1"].tolist(), L["b1"].tolist(), L["U"].tolist(),
                       L["S"].tolist(), L["Vh"].tolist(), L["residuals"].tolist(),
                       L["Wg"].tolist(), L["bg"].tolist())
    rt = O.route(L["x"], L["Wg"], L["bg"])
    free = ~rt["near_tie"]
    y = O.ffn_forward(L["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                      a=np.array(a_b))
    return (np.array_equal(rt["a"][free], np.array(a_b)[free])
            and rel_err(y, np.array(y_b)) <= 1e-12)


@pytest.mark.parametrize("seed,shape", [(0, (23, 16, 64, 4, 16)), (1, (64, 16, 64, 3, 5)),
                                        (2, (1, 16, 64, 1, 16)), (3, (7, 8, 24, 2, 1))])
def test_brute_force_tiny(seed, shape):
    assert check_brute(seed, *shape)


def test_router_exact_integer_ties():
    """Small-integer tokens and router weights make every logit exact; duplicated router rows
    tie and the lower index must win, in the oracle and in the brute force."""
    rng = np.random.default_rng(5)
    x = rng.integers(-3, 4, (64, 16)).astype(float)
    Wg = rng.integers(-2, 3, (4, 16)).astype(float)
    Wg[2] = Wg[1]
    Wg[3] = Wg[0]
    bg = np.zeros(4)
    rt = O.route(x, Wg, bg)
    a_b = [B.token_expert(t, Wg.tolist(), bg.tolist()) for t in x.tolist()]
    assert rt["a"].tolist() == a_b
    assert set(rt["a"].tolist()) <= {0, 1}
    assert rt["near_tie"].all()  # every token has an exact top-2 tie here


# ------------------------------------------------------------------ routing invariants
@pytest.mark.parametrize("E", [1, 2, 5, 8])
def test_routing_invariants(E):
    rng = np.random.default_rng(E)
    T, d = 1000, 24
    x = rng.standard_normal((T, d))
    rt = O.route(x, rng.standard_normal((E, d)), rng.standard_normal(E))
    assert rt["counts"].sum() == T
    assert np.all(np.diff(rt["offsets"]) >= 0) and rt["offsets"][-1] == T
    assert np.array_equal(np.sort(rt["perm"]), np.arange(T))
    keys = rt["a"][rt["perm"]] * T + rt["perm"]
    assert np.all(np.diff(keys) > 0)  # sorted by (expert, token id)
    if E == 1:
        assert np.array_equal(rt["perm"], np.arange(T))


def test_token_permutation_invariance():
    rng = np.random.default_rng(7)
    L = rand_layer(rng, 97, 12, 48, 4, 6)
    y = O.ffn_forward(**{k: L[k] for k in ("x", "W1", "b1", "U", "S", "Vh", "residuals",
                                           "Wg", "bg")})
    p = rng.permutation(97)
    L2 = dict(L, x=L["x"][p])
    y2 = O.ffn_forward(**{k: L2[k] for k in ("x", "W1", "b1", "U", "S", "Vh", "residuals",
                                             "Wg", "bg")})
    assert rel_err(y2, y[p]) <= 1e-14
    r1, r2 = O.route(L["x"], L["Wg"], L["bg"]), O.route(L2["x"], L["Wg"], L["bg"])
    assert np.array_equal(r2["a"], r1["a"][p]) and np.array_equal(r2["counts"], r1["counts"])


def test_token_split_invariance():
    """Tokens are independent: forward(T) = concat(forward(T1), forward(T2)); the routing of
    the whole is the shard routings with offsets added and token ids re-based."""
    rng = np.random.default_rng(8)
    L = rand_layer(rng, 101, 12, 48, 3, 6)
    keys = ("W1", "b1", "U", "S", "Vh", "residuals", "Wg", "bg")
    y = O.ffn_forward(L["x"], *[L[k] for k in keys])
    y1 = O.ffn_forward(L["x"][:40], *[L[k] for k in keys])
    y2 = O.ffn_forward(L["x"][40:], *[L[k] for k in keys])
    assert rel_err(np.concatenate([y1, y2]), y) <= 1e-14
    r, r1, r2 = (O.route(v, L["Wg"], L["bg"]) for v in (L["x"], L["x"][:40], L["x"][40:]))
    assert np.array_equal(r["counts"], r1["counts"] + r2["counts"])
    for e in range(3):
        seg = r["perm"][r["offsets"][e]:r["offsets"][e + 1]]
        s1 = r1["perm"][r1["offsets"][e]:r1["offsets"][e + 1]]
        s2 = r2["perm"][r2["offsets"][e]:r2["offsets"][e + 1]] + 40
        assert np.array_equal(seg, np.concatenate([s1, s2]))


def test_layer_norm_closed_form():
    rng = np.random.default_rng(9)
    y = rng.standard_normal((50, 30)) * 5 + 2
    x = O.layer_norm(y, eps=0.0)
    assert np.allclose(x.mean(1), 0, atol=1e-14) and np.allclose(x.var(1), 1, atol=1e-13)
    assert np.allclose(O.layer_norm(np.array([[1.0, 3.0]]), eps=0.0), [[-1.0, 1.0]])


# ------------------------------------------------------------------ planted mistakes
def _mut_gelu_tanh(u):
    u = np.asarray(u, np.float64)
    return 0.5 * u * (1 + np.tanh(np.sqrt(2 / np.pi) * (u + 0.044715 * u ** 3)))


_ORIG_EXPERTS = O.experts_forward


def _mut_no_unshuffle(z, W_sh, res, a):
    z = O.f64(z)
    srt = O.sort_by_expert(a, len(res))
    out = z @ O.f64(W_sh).T
    zs = z[srt["perm"]]
    for e in range(len(res)):
        lo, hi = srt["offsets"][e], srt["offsets"][e + 1]
        out[lo:hi] += zs[lo:hi] @ O.f64(res[e]).T
    return out


MUTATIONS = {
    "gelu without 1/sqrt2": ("gelu", lambda u: np.asarray(u, float) * 0.5 * (
        1 + __import__("scipy.special").special.erf(np.asarray(u, float)))),
    "gelu tanh form": ("gelu", _mut_gelu_tanh),
    "argmax picks the last maximum": ("argmax_lowest", lambda lg: (
        np.asarray(lg).shape[1] - 1 - np.argmax(np.asarray(lg)[:, ::-1], axis=1))),
    "shared term dropped": ("shared_weight", lambda U, S, Vh: np.zeros(
        (np.shape(U)[0], np.shape(Vh)[1]))),
    "residual term dropped": ("experts_forward", lambda z, W_sh, res, a: O.f64(z) @ O.f64(W_sh).T),
    "no unshuffle": ("experts_forward", _mut_no_unshuffle),
    "every token uses expert 0": ("experts_forward", lambda z, W_sh, res, a: _ORIG_EXPERTS(
        z, W_sh, res, np.zeros_like(np.asarray(a)))),
    "Sigma applied as 1/S": ("shared_weight", lambda U, S, Vh: O.f64(U) @ np.diag(
        1 / O.f64(S)) @ O.f64(Vh)),
    "fold drops the shared term": ("fold_basis", lambda U, S, Vh, res: np.stack(
        [O.f64(R) for R in res])),
    "scale on the shared term too": ("ffn_forward_scaled", lambda x, W1, b1, U, S, Vh, R, s, a=None, **k: (
        O.f64(s)[np.asarray(a)][:, None] * (O.fc1_gelu(x, W1, b1) @ (O.shared_weight(U, S, Vh) + O.f64(R)).T))),
    "router hidden activation dropped": ("relu", lambda u: O.f64(u)),
    "router hidden bias dropped": ("mlp_hidden", lambda x, W_in, b_in, act: O.ROUTER_ACTS[act](
        O.f64(x) @ O.f64(W_in).T)),
    "class tokens routed to experts": ("class_mask", lambda T, s: np.zeros(T, dtype=bool)),
    "fc2 bias added twice": ("fc2_bias", lambda y, b2: O.f64(y) if b2 is None else O.f64(y) + 2 * O.f64(b2)),
    "class token is every token after the first": ("class_mask", lambda T, s: (
        np.arange(T) % s != 0) if s > 0 else np.zeros(T, dtype=bool)),
    "unsorted sub-batches": ("sort_by_expert", lambda a, E: dict(
        a=np.asarray(a), counts=np.bincount(a, minlength=E),
        offsets=np.concatenate([[0], np.cumsum(np.bincount(a, minlength=E))]),
        perm=np.arange(len(a)))),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistakes(name, monkeypatch):
    attr, fake = MUTATIONS[name]
    monkeypatch.setattr(O, attr, fake)
    checks = [check_gelu_table, check_worked_example, check_dense_reduction,
              check_d3_identity, check_scalar_residual, lambda: check_brute(0), check_fold_d3,
              check_folded_brute, check_cls_all_dense, check_cls_brute, check_cls_keeps_routed_rows,
              check_mlp_identity, check_mlp_brute, check_scaled_brute]
    results = []
    for c in checks:
        try:
            results.append(bool(c()))
        except Exception:
            results.append(False)
    assert not all(results), f"no pin caught the planted mistake: {name}"


def test_layernorm_fold_identity():
    """The fold the router and fc1 use for input_layernorm: W LN(y) = rstd (W y - mean W 1), with
    (mean, rstd) the per-row statistics of the oracle's LayerNorm (eps included)."""
    rng = np.random.default_rng(5)
    y = rng.uniform(0.5, 4.0, (64, 1)) * rng.standard_normal((64, 96)) + rng.standard_normal((64, 1))
    W = rng.standard_normal((40, 96))
    mu = y.astype(np.float64).mean(axis=1, keepdims=True)
    rstd = 1.0 / np.sqrt(((y - mu) ** 2).mean(axis=1, keepdims=True) + O.LN_EPS)
    fold = rstd * (y.astype(np.float64) @ W.T - mu * W.sum(axis=1)[None, :])
    assert np.allclose(O.layer_norm(y) @ W.T, fold, rtol=1e-12, atol=1e-10)
