"""GPU parity of the deployment options, through the C ABI: fc2's bias b2 and class tokens on the
dense path (clearmoe_ffn_forward_ex, clearmoe_dense_ffn_forward_ex).

Class tokens (every 197th token from token 0, one per image) skip the router and take the
unconverted fc2, as the paper's dispatch benchmark keeps the class token out of expert dispatch.
Their group follows the experts': idx = E, counts[E] = ceil(T / 197), slots [T - n_cls, T) in
token order. The routed tokens keep the linear router's choice (bit-exact outside near ties),
and every output row is compared with the float64 oracle (ffn_forward_ex) under the layer's
tolerance: the fp32 DeiT-T and bf16 DeiT-S layers in full, the bf16 DeiT-B layer on sampled rows
plus every class row; then the edge cases (all tokens class tokens, T not a multiple of 197, the
1-SM kernels with the slot kernel instead of the fused fc1 epilogue, too many groups)."""
import numpy as np
import pytest
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import Handle, get_routing, handle_for, out_error, sample_rows, tol

pytestmark = pytest.mark.gpu
CLS = 197


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _forward(L, stride, b2=True, T=None):
    s = L["shape"]
    T = s.T if T is None else T
    D = synth.to_torch(L)
    x = D["x"][:T]
    with handle_for(L) as h:
        out = torch.full((T, s.d), float("nan"), device="cuda", dtype=x.dtype)
        cm.clearmoe_ffn_forward_ex(h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                   D["residuals"], D["Wg"], D["bg"], out,
                                   b2=D["b2"] if b2 else None, W2=D["W2"], cls_stride=stride)
        gr = get_routing(h, T, s.E + (1 if stride else 0))
        assert cm.clearmoe_layer_status(h.h) == 0
    return out, gr


def _check_routing(gr, L, stride, T):
    E = L["shape"].E
    x = L["x"][:T]
    rt = O.route_ex(x, L["Wg"], L["bg"], stride)
    free = ~rt["near_tie"]
    bad = int(np.sum(gr["a"][free] != rt["a"][free]))
    assert bad == 0, f"{bad} tokens routed differently (outside near ties)"
    cls = O.class_mask(T, stride)
    assert np.all(gr["a"][cls] == E) and np.all((gr["a"][~cls] >= 0) & (gr["a"][~cls] < E))
    want = O.sort_by_expert(gr["a"], E + (1 if stride else 0))
    assert np.array_equal(gr["counts"], want["counts"]), "counts != histogram of indices"
    assert np.array_equal(gr["offsets"], want["offsets"]), "offsets != prefix sum of counts"
    assert np.array_equal(gr["perm"], want["perm"]), "perm != stable sort by group"
    if stride:
        n_cls = int(cls.sum())
        assert gr["counts"][E] == n_cls and gr["offsets"][E] == T - n_cls
        assert np.array_equal(gr["perm"][T - n_cls:], np.nonzero(cls)[0])


def _oracle(L, rows, a, stride, b2=True):
    """ffn_forward_ex on the given rows: class-ness follows the row's token index."""
    cls = O.class_mask(int(np.max(rows)) + 1, stride)[rows] if stride else np.zeros(len(rows), bool)
    kw = dict(W2=L["W2"], b2=L["b2"] if b2 else None, z_bf16=L["dtype"] == "bf16")
    y = O.ffn_forward_ex(L["x"][rows], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                         a=np.where(cls, 0, a[rows]), **kw)
    if cls.any():  # class rows: the dense path (cls_stride 1 on the sub-batch of class rows)
        y[cls] = O.dense_ffn(L["x"][rows][cls], L["W1"], L["b1"], L["W2"],
                             z_bf16=kw["z_bf16"], b2=kw["b2"])
    return y


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16])
def test_class_tokens_and_b2_full(workload, shape):
    L = workload(shape)
    out, gr = _forward(L, CLS)
    _check_routing(gr, L, CLS, shape.T)
    rows = np.arange(shape.T)
    y = _oracle(L, rows, gr["a"], CLS)
    err = out_error(out, y, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: {err:.3e}"


def test_class_tokens_and_b2_deit_base_sampled(workload):
    L = workload(synth.DEIT_BASE_BF16)
    s = L["shape"]
    out, gr = _forward(L, CLS)
    _check_routing(gr, L, CLS, s.T)
    rows = np.unique(np.concatenate([sample_rows(gr, s.T), np.arange(0, s.T, CLS)]))
    y = _oracle(L, rows, gr["a"], CLS)
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"error {err:.3e}"


def test_b2_alone_and_no_options(workload):
    """b2 without class tokens; and the options at their zero values equal the plain forward."""
    L = workload(synth.DEIT_SMALL_BF16)
    T = L["shape"].T
    out, gr = _forward(L, 0)
    _check_routing(gr, L, 0, T)
    y = _oracle(L, np.arange(T), gr["a"], 0)
    assert out_error(out, y, "bf16") <= tol("bf16")
    plain, _ = _forward(L, 0, b2=False)
    D = synth.to_torch(L)
    with handle_for(L) as h:
        ref = torch.empty_like(plain)
        cm.clearmoe_ffn_forward(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"],
                                D["residuals"], D["Wg"], D["bg"], ref)
        torch.cuda.synchronize()
    assert torch.equal(plain, ref), "zero options change the forward"


@pytest.mark.parametrize("T", [1, 198, 1000])
def test_class_tokens_ragged(workload, T):
    L = workload(synth.DEIT_SMALL_BF16)
    out, gr = _forward(L, CLS, T=T)
    _check_routing(gr, L, CLS, T)
    y = _oracle(L, np.arange(T), gr["a"], CLS)
    assert out_error(out, y, "bf16") <= tol("bf16")


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16, synth.DEIT_BASE_BF16])
def test_every_token_a_class_token_is_the_dense_ffn(workload, shape):
    """No routed rows: no basis launch, so the grouped GEMM follows fc1 directly (DeiT-B: after the
    2-SM basis it would start early; here it must wait for fc1)."""
    L = workload(shape)
    T = min(shape.T, 2000)
    out, gr = _forward(L, 1, T=T)
    assert np.all(gr["a"] == shape.E) and gr["counts"][: shape.E].sum() == 0
    assert np.array_equal(gr["perm"], np.arange(T))
    y = O.dense_ffn(L["x"][:T], L["W1"], L["b1"], L["W2"], z_bf16=L["dtype"] == "bf16", b2=L["b2"])
    err = out_error(out, y, L["dtype"])
    assert err <= tol(L["dtype"]), f"{err:.3e}"


def test_one_sm_kernels_and_slot_kernel():
    """d = 64, H = 320 (no 2-SM tile width divides it): fc1 gathers rows by perm (slot kernel, no
    fused epilogue), the basis and grouped GEMMs run on the 1-SM kernel, whose last group skips the
    t segment."""
    shape = synth.LayerShape("small_1sm_bf16", 1500, 64, 320, 3, 16, "bf16", n_cal=2000)
    L = synth.make_layer(shape)
    out, gr = _forward(L, 50)
    _check_routing(gr, L, 50, shape.T)
    y = _oracle(L, np.arange(shape.T), gr["a"], 50)
    assert out_error(out, y, "bf16") <= tol("bf16")


def test_dense_ffn_with_b2(workload):
    for shape in (synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16):
        L = workload(shape)
        D = synth.to_torch(L)
        T = min(shape.T, 4000)
        with handle_for(L) as h:
            out = torch.full((T, shape.d), float("nan"), device="cuda", dtype=D["x"].dtype)
            cm.clearmoe_dense_ffn_forward_ex(h.h, D["x"][:T], D["W1"], D["b1"], D["W2"], D["b2"], out)
            assert cm.clearmoe_layer_status(h.h) == 0
        y = O.dense_ffn(L["x"][:T], L["W1"], L["b1"], L["W2"], z_bf16=L["dtype"] == "bf16", b2=L["b2"])
        err = out_error(out, y, L["dtype"])
        assert err <= tol(L["dtype"]), f"{shape.name}: {err:.3e}"


def test_option_errors_enqueue_nothing(workload):
    L = workload(synth.DEIT_SMALL_BF16)
    D = synth.to_torch(L)
    s = L["shape"]
    x = D["x"][:256]
    out = torch.zeros(256, s.d, device="cuda", dtype=torch.bfloat16)
    args = (x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"], D["Wg"], D["bg"], out)
    with handle_for(L) as h:
        for kw, code in [(dict(cls_stride=-1, W2=D["W2"]), cm.EINVAL),
                         (dict(cls_stride=CLS, W2=None), cm.EINVAL),
                         (dict(b2=D["b2"][1:]), cm.EINVAL)]:  # b2 not 16-byte aligned
            with pytest.raises(cm.ClearMoEError) as ei:
                cm.clearmoe_ffn_forward_ex(h.h, *args, **kw)
            assert ei.value.code == code
        torch.cuda.synchronize()
        assert torch.count_nonzero(out) == 0
    # sixteen experts leave no group for the class tokens
    with Handle(256, s.d, s.H, 16, s.r, "bf16") as h:
        res = torch.stack([D["residuals"][0]] * 16)
        Wg = torch.cat([D["Wg"]] * 4)
        bg = torch.cat([D["bg"]] * 4)
        with pytest.raises(cm.ClearMoEError) as ei:
            cm.clearmoe_ffn_forward_ex(h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], res, Wg, bg,
                                       out, W2=D["W2"], cls_stride=CLS)
        assert ei.value.code == cm.EUNSUPPORTED


@pytest.mark.parametrize("shape", [synth.DEIT_SMALL_BF16, synth.DEIT_BASE_BF16])
@pytest.mark.parametrize("form", ["folded", "materialized"])
def test_options_on_folded_and_materialized_forms(workload, shape, form):
    """Class tokens and b2 with the basis folded into the experts or materialised, against Eq. 2
    (the oracle's exact W_shared) with the same options: the whole layer at DeiT-S, sampled rows
    plus every class row at DeiT-B."""
    L = workload(shape)
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = torch.full_like(D["x"], float("nan"))
        kw = dict(b2=D["b2"], W2=D["W2"], cls_stride=CLS)
        if form == "folded":
            W = torch.empty_like(D["residuals"])
            cm.clearmoe_fold_basis(h.h, D["U"], D["S"], D["Vh"], D["residuals"], W)
            cm.clearmoe_ffn_forward_folded_ex(h.h, D["x"], D["W1"], D["b1"], W, D["Wg"], D["bg"], out, **kw)
        else:
            W = torch.empty(s.d, s.H, device="cuda", dtype=D["x"].dtype)
            cm.clearmoe_materialize_basis(h.h, D["U"], D["S"], D["Vh"], W)
            cm.clearmoe_ffn_forward_materialized_ex(h.h, D["x"], D["W1"], D["b1"], W, D["residuals"], D["Wg"],
                                                    D["bg"], out, **kw)
        gr = get_routing(h, s.T, s.E + 1)
        assert cm.clearmoe_layer_status(h.h) == 0
    _check_routing(gr, L, CLS, s.T)
    rows = np.arange(s.T) if s.T <= 20000 else np.unique(
        np.concatenate([sample_rows(gr, s.T), np.arange(0, s.T, CLS)]))
    y = _oracle(L, rows, gr["a"], CLS)
    got = out if len(rows) == s.T else out[torch.from_numpy(rows).cuda()]
    err = out_error(got, y, "bf16")
    assert err <= tol("bf16"), f"{form} {s.name}: {err:.3e}"
