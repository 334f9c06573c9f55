"""GPU parity at the limits of the shapes the library accepts, through the C ABI.

E = 16 experts (the largest; the routing kernel's MMA then uses all of its N = 16 columns and the
fused fc1 epilogue's prefix table is full at 152 ranges x 16), d = 1,024 (the largest bf16 width;
the routing kernel's stages then hold four 64-column K blocks, three stages beside W_g's 32 KB,
and H = 4,096 fills fc1's staged bias), and T = max_tokens of the handle. Routing bit-exact outside
near ties, outputs within the bf16 tolerance against the float64 oracle on every row. fp32 layers at
widths where the TF32 tensor-core GEMMs take 128-wide tiles and split K, and at widths that are not
multiples of 16 (the exact-fp32 CUDA-core GEMMs), within the fp32 bound."""
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


def _full_f32(L):
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = run_ffn(h, D)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    y = oracle_rows(L, np.arange(s.T), gr["a"])
    err = out_error(out, y, "f32")
    assert err <= tol("f32"), f"{s.name}: {err:.3e}"
    return err


def test_fp32_tensor_path_wide_tiles():
    """fp32 layer on the TF32 tensor cores at widths where fc1 takes 128-wide tiles and the basis and
    grouped GEMMs split K (d = 384, H = 1,536, E = 8, r = 64, T = 3,000)."""
    _full_f32(synth.make_layer(synth.LayerShape("deit_small_f32", 3000, 384, 1536, 8, 64, "f32",
                                                n_cal=4000)))


def test_fp32_widths_off_sixteen_use_cuda_cores():
    """fp32 widths that are not multiples of 16 (d = 200, r = 12) take the exact-fp32 CUDA-core
    GEMMs; the same parity bound holds."""
    _full_f32(synth.make_layer(synth.LayerShape("d200_f32", 500, 200, 800, 4, 12, "f32",
                                                n_cal=2000)))
