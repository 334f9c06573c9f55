"""GPU parity of the MLP router (Phase 4 "MLP", hidden layer d / 6), through the C ABI.

clearmoe_route_mlp against the oracle's route_mlp: the expert index bit-exact outside near ties
(top-2 float64 logits within 1e-5 relative), counts, offsets and the stable permutation exact, for
the fp32 DeiT-T layer (hidden 32, SIMT), the bf16 DeiT-S layer (hidden 64, 1-SM GEMM) and the bf16
DeiT-B layer (hidden 128, 2-SM GEMM), with ReLU and with GELU; then the whole forward with the MLP
router against the float64 oracle (DeiT-S in full, DeiT-B sampled, with class tokens too)."""
import numpy as np
import pytest
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import get_routing, handle_for, out_error, sample_rows, tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _check(gr, L, M, act):
    E = L["shape"].E
    rt = O.route_mlp(L["x"], M["W_in"], M["b_in"], M["W_out"], M["b_out"], act)
    free = ~rt["near_tie"]
    bad = int(np.sum(gr["a"][free] != rt["a"][free]))
    assert bad == 0, f"{bad} tokens routed differently (outside near ties)"
    want = O.sort_by_expert(gr["a"], E)
    assert np.array_equal(gr["counts"], want["counts"])
    assert np.array_equal(gr["offsets"], want["offsets"])
    assert np.array_equal(gr["perm"], want["perm"])
    return rt


@pytest.mark.parametrize("act", ["relu", "gelu"])
@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16, synth.DEIT_BASE_BF16])
def test_route_mlp(workload, shape, act):
    L = workload(shape)
    M = synth.mlp_router(L, act=act)
    D = synth.to_torch(L | M)
    with handle_for(L) as h:
        m = cm.mlp_router(D["W_in"], D["b_in"], D["W_out"], D["b_out"], act)
        cm.clearmoe_route_mlp(h.h, D["x"], m, shape.E)
        gr = get_routing(h, shape.T, shape.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    rt = _check(gr, L, M, act)
    a_lin = O.route(L["x"], L["Wg"], L["bg"])["a"]
    assert np.mean(rt["a"] == a_lin) > 0.9  # a sensible router


@pytest.mark.parametrize("shape,stride", [(synth.DEIT_SMALL_BF16, 0), (synth.DEIT_SMALL_BF16, 197),
                                          (synth.DEIT_BASE_BF16, 0), (synth.DEIT_TINY_FP32, 197)])
def test_forward_with_mlp_router(workload, shape, stride):
    L = workload(shape)
    M = synth.mlp_router(L, act="gelu")
    D = synth.to_torch(L | M)
    with handle_for(L) as h:
        m = cm.mlp_router(D["W_in"], D["b_in"], D["W_out"], D["b_out"], "gelu")
        out = torch.full_like(D["x"], float("nan"))
        cm.clearmoe_ffn_forward_ex(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   None, None, out, W2=D["W2"] if stride else None, cls_stride=stride,
                                   mlp=m, E=shape.E)
        gr = get_routing(h, shape.T, shape.E + (1 if stride else 0))
        assert cm.clearmoe_layer_status(h.h) == 0
    cls = O.class_mask(shape.T, stride)
    rt = O.route_mlp(L["x"], M["W_in"], M["b_in"], M["W_out"], M["b_out"], "gelu")
    free = ~rt["near_tie"] & ~cls
    assert np.array_equal(gr["a"][free], rt["a"][free]) and np.all(gr["a"][cls] == shape.E)
    rows = np.arange(shape.T) if shape.T <= 20000 else np.unique(np.concatenate(
        [sample_rows(gr, shape.T), np.nonzero(cls)[0]]))
    bf16 = L["dtype"] == "bf16"
    y = O.ffn_forward_ex(L["x"][rows], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"],
                         a=np.where(cls[rows], 0, gr["a"][rows]), z_bf16=bf16)
    if cls[rows].any():
        y[cls[rows]] = O.dense_ffn(L["x"][rows][cls[rows]], L["W1"], L["b1"], L["W2"], z_bf16=bf16)
    got = out if len(rows) == shape.T else out[torch.from_numpy(rows).cuda()]
    err = out_error(got, y, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: {err:.3e}"


def test_mlp_router_argument_errors(workload):
    L = workload(synth.DEIT_SMALL_BF16)
    M = synth.mlp_router(L)
    D = synth.to_torch(L | M)
    x = D["x"][:64]
    with handle_for(L) as h:
        cases = [
            cm.clearmoe_mlp_router(D["W_in"].data_ptr(), D["b_in"].data_ptr(), D["W_out"].data_ptr(),
                                   D["b_out"].data_ptr(), 40, cm.ACT_RELU),   # not a multiple of 16
            cm.clearmoe_mlp_router(D["W_in"].data_ptr(), D["b_in"].data_ptr(), D["W_out"].data_ptr(),
                                   D["b_out"].data_ptr(), 64, 7),             # unknown activation
            cm.clearmoe_mlp_router(D["W_in"].data_ptr(), D["b_in"].data_ptr(), D["W_out"].data_ptr(),
                                   D["b_out"].data_ptr(), 1024, cm.ACT_RELU), # does not fit beside z
            cm.clearmoe_mlp_router(D["W_in"].data_ptr(), None, D["W_out"].data_ptr(),
                                   D["b_out"].data_ptr(), 64, cm.ACT_RELU),   # missing bias
        ]
        for m in cases:
            with pytest.raises(cm.ClearMoEError) as ei:
                cm.clearmoe_route_mlp(h.h, x, m, L["shape"].E)
            assert ei.value.code == cm.EINVAL
