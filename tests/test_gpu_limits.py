"""GPU parity at the limits of the shapes the library accepts, through the C ABI.

E = 16 experts (the largest; the routing kernel's MMA then uses all of its N = 16 columns and the
fused fc1 epilogue's prefix table is full at 152 ranges x 16), d = 1,024 (the largest bf16 width;
the routing kernel's stages then hold four 64-column K blocks, three stages beside W_g's 32 KB,
and H = 4,096 fills fc1's staged bias), and T = max_tokens of the handle. Routing bit-exact outside
near ties, outputs within the bf16 tolerance against the float64 oracle on every row."""
import numpy as np
import pytest
import torch

import synth
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import check_routing, get_routing, handle_for, oracle_rows, out_error, run_ffn, tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _full(L):
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:  # max_tokens = T: the forward runs at the handle's limit
        out = run_ffn(h, D)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    y = oracle_rows(L, np.arange(s.T), gr["a"])
    err = out_error(out, y, "bf16")
    assert err <= tol("bf16"), f"{s.name}: {err:.3e}"
    return gr


def test_sixteen_experts():
    L = synth.make_layer(synth.LayerShape("deit_small_E16", 6000, 384, 1536, 16, 64, "bf16",
                                          n_cal=8000))
    gr = _full(L)
    assert np.count_nonzero(gr["counts"]) >= 12  # most experts receive tokens


def test_widest_layer():
    _full(synth.make_layer(synth.LayerShape("d1024_bf16", 3000, 1024, 4096, 4, 128, "bf16",
                                            n_cal=4000)))
