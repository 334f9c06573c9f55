"""GPU parity at a token count where every routing range spans many 128-row blocks.

The bf16 routing kernel gives each of its 152 CTAs an equal range of tokens and walks it in
128-row blocks, carrying each expert's running count from block to block; a token's word is
expert | rank in the range << 8 (Algorithm 3, "sort z by a": the rank makes the order stable). At
T = 600,000 a range holds 3,948 rows, i.e. 30 full blocks and a partial one, and the ranks run far
past one byte. This file checks: routing bit-exact against the oracle on every token outside near
ties, outputs on a seeded sample plus the whole smallest expert, the handle-free routing entry
point at the same size, whose idx then carries the packed words between its two kernels, and the
router inside fc1, whose slot kernel then spans 4,688 ranges."""
import numpy as np
import pytest
import torch

import synth
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import check_routing, get_routing, handle_for, oracle_rows, out_error, run_ffn, sample_rows, tol

pytestmark = pytest.mark.gpu

T_LARGE = 600_000


@pytest.fixture(scope="module")
def large_layer():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return synth.make_layer(synth.DEIT_BASE_BF16.with_(T=T_LARGE, n_cal=2000, seed=5))


def test_ranges_span_many_blocks():
    """The shape of this file: 152 equal ranges of 3,948 rows, 30 full 128-row blocks and a last
    block of 108 rows (14 boxes of 8 rows, 4 of them past the range's end read and ignored)."""
    chunk = -(-T_LARGE // 152)
    assert chunk == 3948 and chunk // 128 == 30 and chunk % 128 == 108 and -(-108 // 8) * 8 - 108 == 4


def test_forward_at_600k_tokens(large_layer):
    L = large_layer
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = run_ffn(h, D)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    rows = sample_rows(gr, s.T, n=4096, seed=11)
    y = oracle_rows(L, rows, gr["a"][rows])
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"{s.name}: {err:.3e}"


def test_route_noalloc_at_600k_tokens(large_layer):
    L = large_layer
    s = L["shape"]
    D = synth.to_torch(L)
    got = [torch.full((n,), -7, dtype=torch.int32, device="cuda") for n in (s.T, s.E, s.E + 1, s.T)]
    status = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    cm.clearmoe_route_noalloc(D["x"], D["Wg"], D["bg"], *got, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    gr = {k: g.cpu().numpy().astype(np.int64) for k, g in zip(("a", "counts", "offsets", "perm"), got)}
    check_routing(gr, L["x"], L["Wg"], L["bg"])


def test_router_in_fc1_at_600k_tokens(large_layer):
    """The router inside fc1 at the same size: 4,688 ranges of 128 tokens for its slot kernel, routing
    bit-exact on every token outside near ties, outputs on a seeded sample plus the smallest expert."""
    L = large_layer
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = torch.full((s.T, s.d), float("nan"), device="cuda", dtype=torch.bfloat16)
        cm.clearmoe_ffn_forward_ex(h.h, D["x"], D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                                   D["Wg"], D["bg"], out, router_in_fc1=True)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    rows = sample_rows(gr, s.T, n=4096, seed=13)
    y = oracle_rows(L, rows, gr["a"][rows])
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"{s.name} router in fc1: {err:.3e}"
