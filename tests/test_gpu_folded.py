"""GPU parity of the folded form (the shared basis folded into the experts), through the C ABI.

clearmoe_fold_basis against the oracle's float64 fold (within one step of the layer dtype), and
clearmoe_ffn_forward_folded against both the oracle's folded forward on the GPU's own folded
weights and the oracle's unfolded forward (Eq. 2 as the paper states it): the fp32 DeiT-T layer and
the bf16 DeiT-S layer in full, the bf16 DeiT-B layer on sampled rows."""
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


def _fold_and_forward(L):
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        W = torch.empty_like(D["residuals"])
        cm.clearmoe_fold_basis(h.h, D["U"], D["S"], D["Vh"], D["residuals"], W)
        out = torch.full_like(D["x"], float("nan"))
        cm.clearmoe_ffn_forward_folded(h.h, D["x"], D["W1"], D["b1"], W, D["Wg"], D["bg"], out)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    return W, out, gr


def _check_fold(L, W):
    want = O.fold_basis(L["U"], L["S"], L["Vh"], L["residuals"])
    got = W.float().cpu().numpy().astype(np.float64)
    # W_shared accumulated in fp32 over r terms: |error| <= r 2^-23 sum_k |U| |S| |Vh| per element
    r = len(L["S"])
    acc = r * 2.0 ** -23 * (np.abs(L["U"]) @ np.diag(np.abs(L["S"])) @ np.abs(L["Vh"]))
    if L["dtype"] == "bf16":  # then one rounding to bf16: one step of the value
        _, ex = np.frexp(np.abs(want))
        bound = np.ldexp(1.0, ex - 8) + acc[None]
    else:
        bound = np.ldexp(np.abs(want), -23) + acc[None]
    excess = np.abs(got - want) - bound
    assert np.all(excess <= 0), f"fold off by {np.max(excess):.3e} beyond its bound"


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16])
def test_fold_and_folded_forward_full(workload, shape):
    L = workload(shape)
    W, out, gr = _fold_and_forward(L)
    _check_fold(L, W)
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    bf16 = L["dtype"] == "bf16"
    Wd = W.float().cpu().numpy().astype(np.float64)
    y_folded = O.ffn_forward_folded(L["x"], L["W1"], L["b1"], Wd, a=gr["a"], z_bf16=bf16)
    err = out_error(out, y_folded, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: folded weights: {err:.3e}"
    y = oracle_rows(L, np.arange(L["shape"].T), gr["a"])  # Eq. 2 unfolded
    err = out_error(out, y, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: against Eq. 2: {err:.3e}"


def test_folded_forward_deit_base_sampled(workload):
    L = workload(synth.DEIT_BASE_BF16)
    s = L["shape"]
    W, out, gr = _fold_and_forward(L)
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    rows = sample_rows(gr, s.T)
    y = oracle_rows(L, rows, gr["a"][rows])
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"error {err:.3e}"
