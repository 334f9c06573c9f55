"""GPU parity of the input LayerNorm folded into the router and fc1 (input_layernorm), through the
C ABI.

The forward is given the un-normalised stream y (y_t = s_t x_t + m_t, a random scale and shift per
token, rounded to the layer dtype) and must return the sublayer's output on LN(y): the oracle runs
on LN(y) formed in float64 and never rounded, while the GPU never forms LN(y) at all (it applies
W LN(y) = rstd (W y - mean W 1) to its fp32 accumulators). The rules are those of every parity
test: routing bit-exact outside near ties, counts, offsets and the stable permutation exact, and
outputs within the layer's tolerance. Cases: the bf16 DeiT-B layer (2-SM fc1 with the fused slot
epilogue, sampled rows); the fp32 DeiT-T layer in full (SIMT GEMMs, fp32 routing); DeiT-S with
class tokens and b2; the MLP router (bf16 1-SM and 2-SM hidden layers, fp32 SIMT); the 1-SM fc1
that gathers rows by perm (d = 64, H = 320); the folded and materialised bases; the dense FFN;
and the options the dense FFN rejects."""
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


def _streams(L):
    """(device tensors with x = y, the oracle's layer dict with x = LN(y))."""
    y = synth.residual_stream(L["x"], L["dtype"])
    return synth.to_torch(dict(L, x=y)), dict(L, x=O.layer_norm(y))


def _nan_out(T, d, like):
    return torch.full((T, d), float("nan"), device="cuda", dtype=like.dtype)


def _check_out(out, want, dtype, what):
    err = out_error(out, want, dtype)
    assert err <= tol(dtype), f"{what}: {err:.3e}"


@pytest.mark.parametrize("shape", [synth.DEIT_BASE_BF16, synth.DEIT_TINY_FP32],
                         ids=lambda s: s.name)
def test_forward_layernorm_folded(workload, shape):
    L = workload(shape)
    D, Ln = _streams(L)
    with handle_for(L) as h:
        out = _nan_out(shape.T, shape.d, D["x"])
        cm.clearmoe_ffn_forward_ex(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   D["Wg"], D["bg"], out, input_layernorm=True)
        gr = get_routing(h, shape.T, shape.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, Ln["x"], L["Wg"], L["bg"])
    rows = sample_rows(gr, shape.T) if shape.dtype == "bf16" else np.arange(shape.T)
    _check_out(out[torch.from_numpy(rows).cuda()], oracle_rows(Ln, rows, gr["a"][rows]), shape.dtype,
               shape.name)


def test_class_tokens_and_b2(workload):
    shape = synth.DEIT_SMALL_BF16
    L = workload(shape)
    D, Ln = _streams(L)
    T, E, cls = shape.T, shape.E, 197
    with handle_for(L) as h:
        out = _nan_out(T, shape.d, D["x"])
        cm.clearmoe_ffn_forward_ex(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   D["Wg"], D["bg"], out, b2=D["b2"], W2=D["W2"], cls_stride=cls,
                                   input_layernorm=True)
        gr = get_routing(h, T, E + 1)
        assert cm.clearmoe_layer_status(h.h) == 0
    rt = O.route_ex(Ln["x"], L["Wg"], L["bg"], cls)
    free = ~rt["near_tie"]
    assert int(np.sum(gr["a"][free] != rt["a"][free])) == 0
    assert np.array_equal(gr["perm"], O.sort_by_expert(gr["a"], E + 1)["perm"])
    want = O.ffn_forward_ex(Ln["x"], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                            a=np.minimum(gr["a"], E - 1), W2=L["W2"], b2=L["b2"], cls_stride=cls,
                            z_bf16=True)
    _check_out(out, want, "bf16", "class tokens + b2")


@pytest.mark.parametrize("shape,act", [(synth.DEIT_SMALL_BF16, "relu"), (synth.DEIT_BASE_BF16, "gelu"),
                                       (synth.DEIT_TINY_FP32, "gelu")], ids=lambda v: getattr(v, "name", v))
def test_mlp_router(workload, shape, act):
    L = workload(shape)
    M = synth.mlp_router(L, act=act)
    D, Ln = _streams(L)
    Dm = synth.to_torch(dict(M, dtype=L["dtype"]))  # the weights in the layer dtype
    T = min(shape.T, 12608)
    with handle_for(L) as h:
        out = _nan_out(T, shape.d, D["x"])
        m = cm.mlp_router(Dm["W_in"], Dm["b_in"], Dm["W_out"], Dm["b_out"], act)
        cm.clearmoe_ffn_forward_ex(h.h, D["x"][:T], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   None, None, out, mlp=m, E=shape.E, input_layernorm=True)
        gr = get_routing(h, T, shape.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    rt = O.route_mlp(Ln["x"][:T], M["W_in"], M["b_in"], M["W_out"], M["b_out"], act)
    free = ~rt["near_tie"]
    assert int(np.sum(gr["a"][free] != rt["a"][free])) == 0
    assert np.array_equal(gr["perm"], O.sort_by_expert(gr["a"], shape.E)["perm"])
    rows = sample_rows(gr, T, n=2048) if shape.dtype == "bf16" else np.arange(T)
    _check_out(out[torch.from_numpy(rows).cuda()], oracle_rows(Ln, rows, gr["a"][rows]), shape.dtype,
               f"{shape.name} {act}")


def test_gather_fc1_one_sm():
    """d = 64, H = 320: fc1 on the 1-SM kernel, rows gathered by perm, statistics by token."""
    shape = synth.LayerShape("small_1sm_bf16", 1500, 64, 320, 3, 16, "bf16", n_cal=2000)
    L = synth.make_layer(shape)
    D, Ln = _streams(L)
    with handle_for(L) as h:
        out = _nan_out(shape.T, shape.d, D["x"])
        cm.clearmoe_ffn_forward_ex(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   D["Wg"], D["bg"], out, input_layernorm=True)
        gr = get_routing(h, shape.T, shape.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, Ln["x"], L["Wg"], L["bg"])
    _check_out(out, oracle_rows(Ln, np.arange(shape.T), gr["a"]), "bf16", shape.name)


def test_folded_and_materialized_bases(workload):
    shape = synth.DEIT_SMALL_BF16
    L = workload(shape)
    D, Ln = _streams(L)
    T, E = shape.T, shape.E
    with handle_for(L) as h:
        comb = torch.empty_like(D["residuals"])
        cm.clearmoe_fold_basis(h.h, D["U"], D["S"], D["Vh"], D["residuals"], comb)
        W_sh = torch.empty(shape.d, shape.H, device="cuda", dtype=D["x"].dtype)
        cm.clearmoe_materialize_basis(h.h, D["U"], D["S"], D["Vh"], W_sh)
        outs = []
        for form in ("folded", "materialized"):
            out = _nan_out(T, shape.d, D["x"])
            if form == "folded":
                cm.clearmoe_ffn_forward_folded_ex(h.h, D["x"], D["W1"], D["b1"], comb, D["Wg"], D["bg"], out,
                                                  input_layernorm=True)
            else:
                cm.clearmoe_ffn_forward_materialized_ex(h.h, D["x"], D["W1"], D["b1"], W_sh, D["residuals"],
                                                        D["Wg"], D["bg"], out, input_layernorm=True)
            outs.append((form, out, get_routing(h, T, E)))
        assert cm.clearmoe_layer_status(h.h) == 0
    for form, out, gr in outs:
        check_routing(gr, Ln["x"], L["Wg"], L["bg"])
        _check_out(out, oracle_rows(Ln, np.arange(T), gr["a"]), "bf16", form)


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16], ids=lambda s: s.name)
def test_dense_ffn(workload, shape):
    L = workload(shape)
    D, Ln = _streams(L)
    T = min(shape.T, 4000)
    with handle_for(L) as h:
        out = _nan_out(T, shape.d, D["x"])
        cm.clearmoe_dense_ffn_forward_opt(h.h, D["x"][:T], D["W1"], D["b1"], D["W2"], out, b2=D["b2"],
                                          input_layernorm=True)
        assert cm.clearmoe_layer_status(h.h) == 0
    want = O.dense_ffn(Ln["x"][:T], L["W1"], L["b1"], L["W2"], z_bf16=shape.dtype == "bf16", b2=L["b2"])
    _check_out(out, want, shape.dtype, shape.name)


def test_dense_rejects_router_options(workload):
    shape = synth.DEIT_SMALL_BF16
    L = workload(shape)
    D = synth.to_torch(L)
    M = synth.to_torch(dict(synth.mlp_router(L), dtype=L["dtype"]))
    x = D["x"][:256]
    out = torch.zeros(256, shape.d, device="cuda", dtype=x.dtype)
    lib = cm.lib()
    with handle_for(L) as h:
        m = cm.mlp_router(M["W_in"], M["b_in"], M["W_out"], M["b_out"])
        for opt in (cm._options(None, D["W2"], 197, None, True), cm._options(None, None, 0, m, True)):
            rc = lib.clearmoe_dense_ffn_forward_opt(h.h, x.data_ptr(), 256, D["W1"].data_ptr(), D["b1"].data_ptr(),
                                                    D["W2"].data_ptr(), cm.ctypes.byref(opt), out.data_ptr(), None)
            assert rc == cm.EINVAL
        torch.cuda.synchronize()
        assert cm.clearmoe_layer_status(h.h) == 0
    assert torch.count_nonzero(out) == 0  # nothing was enqueued
