"""GPU parity of the one-matrix residual form (Algorithm 2: W_e^res = s_e R), through the C ABI.

clearmoe_ffn_forward_scaled runs every GEMM in token order with the router's choice as a row scale;
its output is compared with the oracle's ffn_forward_scaled (y = W_shared z + s_a R z, float64) on
the GPU's expert choices, which must be bit-exact outside near ties: the fp32 DeiT-T and bf16
DeiT-S layers in full, the bf16 DeiT-B layer on sampled rows; and the routing it leaves behind
(counts, offsets, perm) must be the stable sort of its indices."""
import numpy as np
import pytest
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import check_routing, get_routing, handle_for, out_error, sample_rows, tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16, synth.DEIT_BASE_BF16])
def test_scaled_residual_form(workload, shape):
    L = workload(shape)
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = torch.full_like(D["x"], float("nan"))
        cm.clearmoe_ffn_forward_scaled(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["R"],
                                       D["scales"], D["Wg"], D["bg"], out)
        gr = get_routing(h, shape.T, shape.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    rows = np.arange(shape.T) if shape.T <= 20000 else sample_rows(gr, shape.T)
    s32 = np.asarray(L["scales"], np.float32).astype(np.float64)
    y = O.ffn_forward_scaled(L["x"][rows], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["R"], s32,
                             a=gr["a"][rows], z_bf16=L["dtype"] == "bf16")
    got = out if len(rows) == shape.T else out[torch.from_numpy(rows).cuda()]
    err = out_error(got, y, L["dtype"])
    assert err <= tol(L["dtype"]), f"{shape.name}: {err:.3e}"
