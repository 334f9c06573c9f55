"""GPU parity of the materialised shared basis (the paper's own form of Eq. 2), through the C ABI.

clearmoe_materialize_basis against the oracle's float64 W_shared = U_r diag(S_r) Vh_r (within one
step of the layer dtype plus the fp32 accumulation bound), and clearmoe_ffn_forward_materialized
against the oracle on the GPU's own W_sh and against Eq. 2 with the exact W_shared: the fp32 DeiT-T
and bf16 DeiT-S layers in full, the bf16 DeiT-B layer on sampled rows."""
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


def _materialize_and_forward(L):
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        W = torch.empty(s.d, s.H, device="cuda", dtype=D["x"].dtype)
        cm.clearmoe_materialize_basis(h.h, D["U"], D["S"], D["Vh"], W)
        out = torch.full_like(D["x"], float("nan"))
        cm.clearmoe_ffn_forward_materialized(h.h, D["x"], D["W1"], D["b1"], W, D["residuals"], D["Wg"],
                                             D["bg"], out)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    return W, out, gr


def _check_basis(L, W):
    want = O.shared_weight(L["U"], L["S"], L["Vh"])
    got = W.float().cpu().numpy().astype(np.float64)
    r = len(L["S"])
    acc = r * 2.0 ** -23 * (np.abs(L["U"]) @ np.diag(np.abs(L["S"])) @ np.abs(L["Vh"]))
    if L["dtype"] == "bf16":
        _, ex = np.frexp(np.abs(want))
        bound = np.ldexp(1.0, ex - 8) + acc
    else:
        bound = np.ldexp(np.abs(want), -23) + acc
    excess = np.abs(got - want) - bound
    assert np.all(excess <= 0), f"W_sh off by {np.max(excess):.3e} beyond its bound"


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16])
def test_materialized_full(workload, shape):
    L = workload(shape)
    W, out, gr = _materialize_and_forward(L)
    _check_basis(L, W)
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    bf16 = L["dtype"] == "bf16"
    z = O.fc1_gelu(L["x"], L["W1"], L["b1"], z_bf16=bf16)
    y_gpu_w = O.experts_forward(z, W.float().cpu().numpy().astype(np.float64), L["residuals"], gr["a"])
    err = out_error(out, y_gpu_w, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: on the GPU's W_sh: {err:.3e}"
    y = oracle_rows(L, np.arange(shape.T), gr["a"])  # Eq. 2 with the exact W_shared
    err = out_error(out, y, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: against Eq. 2: {err:.3e}"


def test_materialized_deit_base_sampled(workload):
    L = workload(synth.DEIT_BASE_BF16)
    s = L["shape"]
    W, out, gr = _materialize_and_forward(L)
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    rows = sample_rows(gr, s.T)
    y = oracle_rows(L, rows, gr["a"][rows])
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"error {err:.3e}"
