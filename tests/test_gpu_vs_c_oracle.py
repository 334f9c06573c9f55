"""GPU parity against the plain-C oracle (oracle/clearmoe_ref.c), through the C ABI.

The same rules as the other parity tests, with the C restatement of the layer as the reference:
the expert index bit-exact except where the C oracle's float64 top-2 logits are within 1e-5
relative of each other, counts / offsets / perm exactly the stable sort of the GPU's indices, and
the outputs (on the GPU's expert choice) within the layer's tolerance. The fp32 DeiT-T layer is
checked in full, the bf16 DeiT-S layer on a seeded sample of rows plus one whole expert.
`check_against_c_oracle` is also run on the CPU (tests/test_oracle_c.py) with the numpy oracle's
output in place of the GPU's."""
import numpy as np
import pytest
import torch

import synth
from oracle import ref_c as C
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import get_routing, handle_for, run_ffn

pytestmark = pytest.mark.gpu

NEAR_TIE_REL = 1e-5
TOL = {"f32": 1e-4, "bf16": 2e-2}


def check_against_c_oracle(L: dict, out: np.ndarray, gr: dict, rows=None) -> float:
    """Asserts the routing rules against the C oracle's routing; returns the output error of the
    given rows (all when None) against the C oracle's forward on the GPU's expert choice."""
    E = np.asarray(L["Wg"]).shape[0]
    lg = C.router_logits(L["x"], L["Wg"], L["bg"])
    top = np.sort(lg, axis=1)[:, -2:]
    near = (top[:, 1] - top[:, 0]) <= NEAR_TIE_REL * np.maximum(np.abs(top[:, 0]), np.abs(top[:, 1]))
    a_c = C.argmax(lg)
    bad = int(np.sum(gr["a"][~near] != a_c[~near]))
    assert bad == 0, f"{bad} tokens routed differently from the C oracle (outside near ties)"
    srt = C.sort_by_group(gr["a"], E)
    for k in ("counts", "offsets", "perm"):
        assert np.array_equal(gr[k], srt[k]), k
    rows = np.arange(L["x"].shape[0]) if rows is None else np.asarray(rows)
    y = C.ffn_forward(L["x"][rows], L["W1"], L["b1"], L["U"], L["S"], L["Vh"], L["residuals"], gr["a"][rows],
                      z_bf16=L["dtype"] == "bf16")
    g = np.asarray(out, np.float64)[rows]
    assert np.all(np.isfinite(g)), "non-finite outputs"
    if L["dtype"] == "bf16":
        return float(np.abs(g - y).max() / np.sqrt(np.mean(y ** 2)))
    return float(np.linalg.norm(g - y) / np.linalg.norm(y))


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


@pytest.mark.parametrize("shape", [synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16], ids=lambda s: s.name)
def test_layer_against_c_oracle(workload, shape):
    L = workload(shape)
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = run_ffn(h, D)
        gr = get_routing(h, shape.T, shape.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    rows = None
    if shape.dtype == "bf16":  # a seeded sample plus every row of the smallest non-empty expert
        rng = np.random.default_rng(0)
        nz = np.nonzero(gr["counts"])[0]
        small = np.nonzero(gr["a"] == nz[np.argmin(gr["counts"][nz])])[0]
        rows = np.unique(np.concatenate([rng.choice(shape.T, 512, replace=False), small[:512]]))
    err = check_against_c_oracle(L, out.float().cpu().numpy(), gr, rows)
    assert err <= TOL[shape.dtype], f"{shape.name}: {err:.3e}"
