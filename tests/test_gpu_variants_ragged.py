"""Every forward variant at ragged token counts (T = 1, 17, 300 on the DeiT-S bf16 layer), through
the C ABI, against the float64 oracle: the folded and materialised basis forms, the one-residual-
matrix form, the MLP router and the folded input LayerNorm (the forward given y, the oracle run on
LN(y)). A single token, a token count below one 16-row routing stage and
one that leaves a partial 256-row tile all run the same kernels as the full layer."""
import numpy as np
import pytest
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import get_routing, handle_for, out_error, tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


@pytest.mark.parametrize("T", [1, 17, 300])
@pytest.mark.parametrize("form", ["folded", "materialized", "scaled", "mlp", "layernorm"])
def test_variant_ragged(workload, form, T):
    L = workload(synth.DEIT_SMALL_BF16)
    s = L["shape"]
    M = synth.mlp_router(L, act="relu")
    D = synth.to_torch(L | M)
    x = D["x"][:T]
    y = synth.residual_stream(L["x"], "bf16")[:T]  # the un-normalised stream of the LayerNorm form
    with handle_for(L) as h:
        out = torch.full((T, s.d), float("nan"), device="cuda", dtype=torch.bfloat16)
        if form == "folded":
            W = torch.empty_like(D["residuals"])
            cm.clearmoe_fold_basis(h.h, D["U"], D["S"], D["Vh"], D["residuals"], W)
            cm.clearmoe_ffn_forward_folded(h.h, x, D["W1"], D["b1"], W, D["Wg"], D["bg"], out)
        elif form == "materialized":
            W = torch.empty(s.d, s.H, device="cuda", dtype=torch.bfloat16)
            cm.clearmoe_materialize_basis(h.h, D["U"], D["S"], D["Vh"], W)
            cm.clearmoe_ffn_forward_materialized(h.h, x, D["W1"], D["b1"], W, D["residuals"], D["Wg"], D["bg"], out)
        elif form == "scaled":
            cm.clearmoe_ffn_forward_scaled(h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["R"],
                                           D["scales"], D["Wg"], D["bg"], out)
        elif form == "layernorm":
            yd = synth.to_torch({"x": y, "dtype": "bf16"})["x"]
            cm.clearmoe_ffn_forward_ex(h.h, yd, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                       D["Wg"], D["bg"], out, input_layernorm=True)
        else:
            m = cm.mlp_router(D["W_in"], D["b_in"], D["W_out"], D["b_out"], "relu")
            cm.clearmoe_ffn_forward_ex(h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                       None, None, out, mlp=m, E=s.E)
        gr = get_routing(h, T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    xs = O.layer_norm(y) if form == "layernorm" else L["x"][:T]
    if form == "mlp":
        rt = O.route_mlp(xs, M["W_in"], M["b_in"], M["W_out"], M["b_out"], "relu")
    else:
        rt = O.route(xs, L["Wg"], L["bg"])
    free = ~rt["near_tie"]
    assert np.array_equal(gr["a"][free], rt["a"][free])
    assert np.array_equal(gr["perm"], O.sort_by_expert(gr["a"], s.E)["perm"])
    if form == "scaled":
        s32 = np.asarray(L["scales"], np.float32).astype(np.float64)
        y = O.ffn_forward_scaled(xs, L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["R"], s32, a=gr["a"],
                                 z_bf16=True)
    else:  # Eq. 2 with the exact W_shared: the folded and materialised forms round it once more
        y = O.ffn_forward(xs, L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], a=gr["a"], z_bf16=True)
    err = out_error(out, y, "bf16")
    assert err <= tol("bf16"), f"{form} T={T}: {err:.3e}"
