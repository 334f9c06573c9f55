"""GPU parity of the router inside fc1 (clearmoe_ffn_options.router_in_fc1), through the C ABI.

fc1's kernel computes the linear router's logits W_g x + b_g (Phase 4 "Linear"; Algorithm 3 step 3)
from the token tiles it loads for fc1 and takes the argmax (lowest index on ties) in its epilogue;
the slots come from per-128-token-range counts and ranks ("sort z by a", stable), the basis factor
stores t at each token's slot and the grouped GEMM gathers z rows by perm. Checked against the
float64 oracle under the same rules as the default path (routing bit-exact outside near ties,
counts / offsets / perm the stable sort of the GPU's indices, outputs within the bf16 tolerance),
and against the default path itself: where both paths pick the same expert for every token the
outputs are bitwise equal (same z rows, same slots, same tiles)."""
import numpy as np
import pytest
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import check_routing, get_routing, handle_for, oracle_rows, out_error, sample_rows, tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _forward(h, D, T, fused, folded_W=None):
    x = D["x"][:T]
    out = torch.full((T, D["W1"].shape[1]), float("nan"), device="cuda", dtype=x.dtype)
    if folded_W is not None:
        cm.clearmoe_ffn_forward_folded_ex(h.h, x, D["W1"], D["b1"], folded_W, D["Wg"], D["bg"], out,
                                          router_in_fc1=fused)
    else:
        cm.clearmoe_ffn_forward_ex(h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   D["Wg"], D["bg"], out, router_in_fc1=fused)
    return out


def _check(L, T=None, rows=None, folded=False):
    s = L["shape"]
    T = s.T if T is None else T
    D = synth.to_torch(L)
    with handle_for(L) as h:
        W = None
        if folded:
            W = torch.empty_like(D["residuals"])
            cm.clearmoe_fold_basis(h.h, D["U"], D["S"], D["Vh"], D["residuals"], W)
        ref = _forward(h, D, T, False, W).clone()
        gref = get_routing(h, T, s.E)
        out = _forward(h, D, T, True, W)
        gr = get_routing(h, T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    x = L["x"][:T]
    check_routing(gr, x, L["Wg"], L["bg"])
    if np.array_equal(gr["a"], gref["a"]):  # same experts everywhere: the same arithmetic
        assert torch.equal(out, ref), "outputs differ from the default path with identical routing"
    if rows is None:
        rows = np.arange(T)
    if folded:  # the oracle's folded forward on the GPU's folded weights (their bf16 rounding is the fold's)
        Wc = W.float().cpu().numpy().astype(np.float64)
        y = O.ffn_forward_folded(x[rows], L["W1"], L["b1"], Wc, a=gr["a"][rows], z_bf16=True)
    else:
        y = oracle_rows(dict(L, x=x), rows, gr["a"][rows])
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"{s.name} T={T}: {err:.3e}"
    return gr


def test_deit_small_full(workload):
    """DeiT-S (r = 64: the 1-SM basis kernel stores t at the slots)."""
    _check(workload(synth.DEIT_SMALL_BF16))


def test_deit_base_sampled(workload):
    L = workload(synth.DEIT_BASE_BF16)
    D = synth.to_torch(L)
    with handle_for(L) as h:
        _forward(h, D, L["shape"].T, True)
        gr = get_routing(h, L["shape"].T, L["shape"].E)
    _check(L, rows=sample_rows(gr, L["shape"].T, n=4096, seed=3))


@pytest.mark.parametrize("T", [1, 17, 127, 128, 129, 300, 1000])
def test_ragged_token_counts(workload, T):
    """Partial 128-token ranges, a single token, and a partial 256-token pair tile."""
    _check(workload(synth.DEIT_SMALL_BF16), T=T)


def test_folded_basis(workload):
    _check(workload(synth.DEIT_SMALL_BF16), folded=True)
    _check(workload(synth.DEIT_SMALL_BF16), T=300, folded=True)


def test_sixteen_experts_and_empty_ones():
    """E = 16 (the router unit's full 16 columns) with two experts that never win."""
    L = synth.make_layer(synth.LayerShape("deit_small_E16", 5000, 384, 1536, 16, 64, "bf16", n_cal=8000))
    bg = L["bg"].copy()
    bg[[3, 9]] = -1e4
    gr = _check(dict(L, bg=synth.round_bf16(bg)))
    assert gr["counts"][3] == 0 and gr["counts"][9] == 0


def test_exact_ties_take_lowest_index():
    """Integer tokens and router rows: every logit exact in fp32, duplicated rows tie, the lower
    index wins bit-exactly in the fc1 epilogue's argmax too."""
    rng = np.random.default_rng(11)
    L = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=600, E=4, n_cal=2000))
    x = rng.integers(-3, 4, (600, 384)).astype(np.float32)
    Wg = rng.integers(-2, 3, (4, 384)).astype(np.float32)
    Wg[3] = Wg[1]
    Wg[2] = Wg[0]
    L = dict(L, x=x, Wg=Wg, bg=np.zeros(4, np.float32))
    D = synth.to_torch(L)
    with handle_for(L) as h:
        _forward(h, D, 600, True)
        gr = get_routing(h, 600, 4)
        assert cm.clearmoe_layer_status(h.h) == 0
    want = O.sort_by_expert(O.argmax_lowest(O.router_logits(x, Wg, np.zeros(4))), 4)
    assert np.array_equal(gr["a"], want["a"]) and set(gr["a"].tolist()) <= {0, 1}
    assert np.array_equal(gr["perm"], want["perm"])
    assert np.array_equal(gr["counts"], want["counts"])


def test_unsupported_combinations(workload):
    L = workload(synth.DEIT_SMALL_BF16)
    D = synth.to_torch(L)
    M = synth.to_torch(synth.mlp_router(L) | {"dtype": "bf16"})
    mlp = cm.mlp_router(M["W_in"], M["b_in"], M["W_out"], M["b_out"], "relu")
    with handle_for(L) as h:
        out = torch.zeros(100, 384, device="cuda", dtype=torch.bfloat16)
        x = D["x"][:100]
        args = (h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"])
        for kw in (dict(cls_stride=197, W2=D["W2"]), dict(input_layernorm=True)):
            with pytest.raises(cm.ClearMoEError) as e:
                cm.clearmoe_ffn_forward_ex(*args, D["Wg"], D["bg"], out, router_in_fc1=True, **kw)
            assert e.value.code == cm.EUNSUPPORTED
        with pytest.raises(cm.ClearMoEError) as e:
            cm.clearmoe_ffn_forward_ex(*args, None, None, out, mlp=mlp, E=4, router_in_fc1=True)
        assert e.value.code == cm.EUNSUPPORTED
        torch.cuda.synchronize()
        assert torch.count_nonzero(out) == 0
    Lt = workload(synth.DEIT_TINY_FP32)
    Dt = synth.to_torch(Lt)
    with handle_for(Lt) as h:
        out = torch.zeros(50, 192, device="cuda")
        with pytest.raises(cm.ClearMoEError) as e:
            cm.clearmoe_ffn_forward_ex(h.h, Dt["x"][:50], Dt["W1"], Dt["b1"], Dt["U"], Dt["S"], Dt["Vh"],
                                       Dt["residuals"], Dt["Wg"], Dt["bg"], out, router_in_fc1=True)
        assert e.value.code == cm.EUNSUPPORTED


def test_single_expert_is_token_order():
    """E = 1: every token takes expert 0 and the permutation is the identity."""
    L = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=777, E=1, n_cal=2000))
    gr = _check(L)
    assert np.array_equal(gr["perm"], np.arange(777)) and np.all(gr["a"] == 0)


def test_widest_layer():
    """d = 1,024 (16 K blocks in the router unit) and H = 4,096 (the widest fc1 the 2-SM kernel
    stages a bias for)."""
    _check(synth.make_layer(synth.LayerShape("d1024_bf16", 3000, 1024, 4096, 4, 128, "bf16", n_cal=4000)))
