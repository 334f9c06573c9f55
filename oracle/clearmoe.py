"""Float64 oracle of one CLEAR-MoE FFN layer (test infrastructure; see the package docstring).

Notation follows the paper: tokens x [T x d], fc1 W1 [H x d] + b1 [H], z = GELU(fc1(x)) [T x H],
fc2 W2 [d x H], truncated SVD W_shared = U_r Sigma_r V_r^T with U_r [d x r], Sigma_r = diag(S_r),
V_r^T = Vh_r [r x H], residual experts W_e^res [d x H], linear router W_g [E x d], b_g [E].

Every step is taken in the order of Algorithm 3:
  1. z <- GELU(fc1(x))                      (shared, all tokens)
  2. h_sh <- z W_shared^T                    (W_shared materialised, as the paper does)
  3. a <- argmax(g(x))                       (top-1 expert assignment)
  4. sort z by a; sub-batch boundaries       (stable sort; counts and offsets)
  5. h_res[e] <- z_e (W_e^res)^T             (one product per expert sub-batch)
  6. unshuffle h_res; y <- h_sh + h_res
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

NEAR_TIE_REL = 1e-5  # router-logit top-2 gap below which a token's expert is not compared
LN_EPS = 1e-6


def f64(a) -> np.ndarray:
    return np.asarray(a, dtype=np.float64)


# ---------------------------------------------------------------- quantisation point (bf16)
def to_bf16(v) -> np.ndarray:
    """Round float64 values to the nearest bf16 (8 significant bits), ties to even.

    v = m * 2**e with 0.5 <= |m| < 1 (frexp); bf16 keeps 8 bits of m, so the result is
    rint(m * 2**8) * 2**(e - 8), and numpy's rint rounds halves to even."""
    m, e = np.frexp(f64(v))
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


# ---------------------------------------------------------------- Phase 4 router + Alg. 3 step 3
def router_logits(x, Wg, bg, precision=np.float64) -> np.ndarray:
    """Linear router g(x) = W_g x + b_g (Section "Phase 4: Router Fitting", Linear router with
    d x E weights and a bias per expert)."""
    x, Wg, bg = (np.asarray(a, dtype=precision) for a in (x, Wg, bg))
    return x @ Wg.T + bg


def relu(u) -> np.ndarray:
    return np.maximum(f64(u), 0.0)


ROUTER_ACTS = {"relu": lambda u: relu(u), "gelu": lambda u: gelu(u)}


def mlp_hidden(x, W_in, b_in, act: str) -> np.ndarray:
    """The MLP router's hidden layer act(W_in x + b_in), float64."""
    return ROUTER_ACTS[act](f64(x) @ f64(W_in).T + f64(b_in))


def mlp_router_logits(x, W_in, b_in, W_out, b_out, act: str = "relu", precision=np.float64):
    """MLP router g(x) = W_out act(W_in x + b_in) + b_out (Phase 4, "MLP": one hidden layer of d/6
    units; the paper does not name the activation, both ReLU and GELU are offered). With
    precision float32 the hidden layer is formed in float64, stored in float32, and the output
    layer is evaluated in float32 (the precision of the decision)."""
    h = mlp_hidden(x, W_in, b_in, act)
    h, W_out, b_out = (np.asarray(a, dtype=precision) for a in (h, W_out, b_out))
    return h @ W_out.T + b_out


def route_mlp(x, W_in, b_in, W_out, b_out, act: str = "relu") -> dict:
    """Algorithm 3 steps 3-4 with the MLP router: the decision on float32 logits, near ties
    flagged from float64 logits as for the linear router."""
    E = np.asarray(W_out).shape[0]
    a = argmax_lowest(mlp_router_logits(x, W_in, b_in, W_out, b_out, act, precision=np.float32))
    lg = mlp_router_logits(x, W_in, b_in, W_out, b_out, act)
    return sort_by_expert(a, E) | dict(near_tie=_near_tie_logits(lg))


def argmax_lowest(logits) -> np.ndarray:
    """a_t = min{e : logit_{t,e} = max_e logit_{t,e}} (Algorithm 3, "a <- argmax g(x)"; the
    paper leaves ties open, the lowest index wins here)."""
    return np.argmax(logits, axis=1).astype(np.int64)  # numpy returns the first maximum


def near_ties(x, Wg, bg, rel=NEAR_TIE_REL) -> np.ndarray:
    """Tokens whose top-2 router logits (float64) differ by less than rel * max(|l1|, |l2|)."""
    return _near_tie_logits(router_logits(x, Wg, bg), rel)


def _near_tie_logits(lg, rel=NEAR_TIE_REL) -> np.ndarray:
    if lg.shape[1] < 2:
        return np.zeros(lg.shape[0], dtype=bool)
    top = np.sort(lg, axis=1)[:, -2:]
    gap = top[:, 1] - top[:, 0]
    scale = np.maximum(np.abs(top[:, 0]), np.abs(top[:, 1]))
    return gap <= rel * scale


def route(x, Wg, bg) -> dict:
    """Algorithm 3 steps 3-4: expert index per token, then "sort z by a" with sub-batch
    boundaries. The decision is taken on float32 logits (the precision the router is run in);
    the sort is stable (ascending token id within an expert)."""
    E = np.asarray(Wg).shape[0]
    a = argmax_lowest(router_logits(x, Wg, bg, precision=np.float32))
    return sort_by_expert(a, E) | dict(near_tie=near_ties(x, Wg, bg))


def sort_by_expert(a, E: int) -> dict:
    """counts_e = |{t : a_t = e}|, offsets = exclusive prefix sum (E + 1 entries),
    perm[slot] = token, tokens of expert e in slots [offsets_e, offsets_{e+1}) in id order."""
    a = np.asarray(a, dtype=np.int64)
    counts = np.bincount(a, minlength=E).astype(np.int64)
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)
    perm = np.argsort(a, kind="stable").astype(np.int64)
    return dict(a=a, counts=counts, offsets=offsets, perm=perm)


# ---------------------------------------------------------------- Eq. 2 pieces
def gelu(u) -> np.ndarray:
    """GELU(u) = u * Phi(u), Phi the standard normal CDF = (1 + erf(u / sqrt 2)) / 2."""
    u = f64(u)
    return u * 0.5 * (1.0 + erf(u / np.sqrt(2.0)))


def fc1_gelu(x, W1, b1, z_bf16: bool = False) -> np.ndarray:
    """z = GELU(fc1(x)) = GELU(x W1^T + b1) (Eq. 2; Algorithm 3 step 1). With z_bf16 the
    hidden state is stored in bf16, as the bf16 layer stores it."""
    z = gelu(f64(x) @ f64(W1).T + f64(b1))
    return to_bf16(z) if z_bf16 else z


def shared_weight(U, S, Vh) -> np.ndarray:
    """W_shared = U_r Sigma_r V_r^T, materialised as a dense d x H matrix (Eq. 2 and the
    Phase 3 text: materialised before inference, no factorised compute)."""
    return f64(U) @ np.diag(f64(S)) @ f64(Vh)


def experts_forward(z, W_sh, residuals, a) -> np.ndarray:
    """Algorithm 3 steps 2 and 4-6 on hidden states z [T x H] with assignment a [T]."""
    z = f64(z)
    T = z.shape[0]
    E = len(residuals)
    h_sh = z @ f64(W_sh).T                                   # step 2
    srt = sort_by_expert(a, E)                               # step 4
    z_sorted = z[srt["perm"]]
    h_res_sorted = np.zeros((T, f64(W_sh).shape[0]))
    for e in range(E):                                       # step 5
        lo, hi = srt["offsets"][e], srt["offsets"][e + 1]
        if hi > lo:
            h_res_sorted[lo:hi] = z_sorted[lo:hi] @ f64(residuals[e]).T
    h_res = np.empty_like(h_res_sorted)
    h_res[srt["perm"]] = h_res_sorted                        # step 6: unshuffle
    return h_sh + h_res


def ffn_forward(x, W1, b1, U, S, Vh, residuals, Wg=None, bg=None, a=None,
                z_bf16: bool = False) -> np.ndarray:
    """y = W_shared z + W_{a}^res z, z = GELU(fc1(x)) (Eq. 2 / Algorithm 3). `a` overrides the
    router's assignment (random routing, or the near-tie substitution of the parity tests)."""
    if a is None:
        a = route(x, Wg, bg)["a"]
    z = fc1_gelu(x, W1, b1, z_bf16)
    return experts_forward(z, shared_weight(U, S, Vh), residuals, a)


def ffn_forward_scaled(x, W1, b1, U, S, Vh, R, s, Wg=None, bg=None, a=None,
                       z_bf16: bool = False) -> np.ndarray:
    """Eq. 2 with the residual structure of Algorithm 2, W_e^res = s_e (W2 - W_shared) = s_e R:
    y_t = W_shared z_t + s_{a_t} R z_t (one residual matrix and a scalar per expert)."""
    if a is None:
        a = route(x, Wg, bg)["a"]
    z = fc1_gelu(x, W1, b1, z_bf16)
    return z @ shared_weight(U, S, Vh).T + f64(s)[np.asarray(a)][:, None] * (z @ f64(R).T)


def fold_basis(U, S, Vh, residuals) -> np.ndarray:
    """W_e^comb = W_shared + W_e^res for every expert e: Eq. 2 regrouped, since both terms act
    on the same hidden state, y = W_shared z + W_a^res z = (W_shared + W_a^res) z."""
    W_sh = shared_weight(U, S, Vh)
    return np.stack([W_sh + f64(R) for R in residuals])


def ffn_forward_folded(x, W1, b1, W_comb, Wg=None, bg=None, a=None,
                       z_bf16: bool = False) -> np.ndarray:
    """y = W_comb[a] z, z = GELU(fc1(x)): Algorithm 3 on folded weights (no shared step 2;
    steps 4-6 with W_comb in place of the residuals)."""
    if a is None:
        a = route(x, Wg, bg)["a"]
    z = fc1_gelu(x, W1, b1, z_bf16)
    return experts_forward(z, np.zeros((f64(W_comb[0]).shape[0], z.shape[1])), W_comb, a)


def dense_ffn(x, W1, b1, W2, z_bf16: bool = False, b2=None) -> np.ndarray:
    """The unconverted layer: y = W2 GELU(W1 x + b1) (the dense FFN, D0), + b2 when given."""
    return fc2_bias(fc1_gelu(x, W1, b1, z_bf16) @ f64(W2).T, b2)


# ---------------------------------------------------------------- deployment: fc2 bias, class tokens
def fc2_bias(y, b2) -> np.ndarray:
    """y + b2 on every row: the fc2 bias of the pretrained layer, which Eq. 2 leaves out (a bias
    is unchanged by the SVD split of W2, so it is added once per token, outside both terms)."""
    return f64(y) if b2 is None else f64(y) + f64(b2)


def class_mask(T: int, cls_stride: int) -> np.ndarray:
    """Class tokens among T: token t with t % cls_stride == 0 (the class token leads each image's
    cls_stride tokens, 197 for a ViT at 224 px, patch 16); none when cls_stride is 0."""
    t = np.arange(T)
    return t % cls_stride == 0 if cls_stride > 0 else np.zeros(T, dtype=bool)


def route_ex(x, Wg, bg, cls_stride: int = 0) -> dict:
    """Routing with the class token kept out of expert dispatch and run on the dense path (the
    dispatch micro-benchmark table, appendix "Dispatch Benchmark and Parallel Scaling", excludes
    it from dispatch and processes it on the dense path): class tokens skip the router and
    form group E, placed after every expert's group, in token order (counts: E + 1 entries,
    offsets: E + 2)."""
    E = np.asarray(Wg).shape[0]
    rt = route(x, Wg, bg)
    cls = class_mask(len(rt["a"]), cls_stride)
    a = np.where(cls, E, rt["a"])
    return sort_by_expert(a, E + (1 if cls_stride > 0 else 0)) | dict(near_tie=rt["near_tie"] & ~cls)


def ffn_forward_ex(x, W1, b1, U, S, Vh, residuals, Wg=None, bg=None, a=None, W2=None, b2=None,
                   cls_stride: int = 0, z_bf16: bool = False) -> np.ndarray:
    """Eq. 2 as deployed: a routed token gets y_t = W_shared z_t + W_{a_t}^res z_t + b2, a class
    token y_t = W2 z_t + b2 (the unconverted fc2, the dense path). `a` as in ffn_forward (its
    entries for class tokens are not used)."""
    if a is None:
        a = route(x, Wg, bg)["a"]
    z = fc1_gelu(x, W1, b1, z_bf16)
    cls = class_mask(z.shape[0], cls_stride)
    y = experts_forward(z, shared_weight(U, S, Vh), residuals, np.where(cls, 0, a))
    if cls.any():
        y[cls] = z[cls] @ f64(W2).T
    return fc2_bias(y, b2)


# ---------------------------------------------------------------- the 12-sublayer stack
def layer_norm(y, eps: float = LN_EPS) -> np.ndarray:
    """Per-token LayerNorm without affine: (y - mean) / sqrt(biased variance + eps)."""
    y = f64(y)
    mu = y.mean(axis=1, keepdims=True)
    var = ((y - mu) ** 2).mean(axis=1, keepdims=True)
    return (y - mu) / np.sqrt(var + eps)


def stack_layer(x, L: dict, a=None, bf16: bool = True) -> np.ndarray:
    """One sublayer of the stack: CLEAR-MoE FFN or dense FFN, output stored in bf16."""
    if L["moe"]:
        y = ffn_forward(x, L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                        L["Wg"], L["bg"], a=a, z_bf16=bf16)
    else:
        y = dense_ffn(x, L["W1"], L["b1"], L["W2"], z_bf16=bf16)
    return to_bf16(y) if bf16 else y


def stack_next_input(y, bf16: bool = True) -> np.ndarray:
    """x_{l+1} = LN(y_l), stored in bf16."""
    x = layer_norm(y)
    return to_bf16(x) if bf16 else x
