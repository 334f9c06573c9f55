"""GPU parity at a token count where the routing kernel keeps its per-row words in global memory.

The routing kernel stores each of its rows' words (expert | rank in the range) and per-stage
expert counts in shared memory while they fit beside W_g and the eight-stage copy ring. At the
DeiT-B width (d = 768, bf16, E = 8) that space holds about 2,620 rows per CTA, so above ~398 K
tokens (152 CTAs) the words go to idx in global memory and the ranks come from the match-mask loop
instead of the per-stage ballots (Algorithm 3, "sort z by a": the same stable order either way).
This file runs that path at T = 600,000 (3,948 rows per CTA): routing bit-exact against the oracle
on every token outside near ties, outputs on a seeded sample plus the whole smallest expert, the
handle-free routing entry point at the same size, whose idx then carries the packed words between
its two kernels, and the router inside fc1, whose slot kernel then spans 4,688 ranges."""
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


def test_rows_per_cta_exceed_shared_memory():
    """The shape of this file is past the shared-memory limit of the per-row words: 152 equal
    ranges of 3,948 rows need 3,948 x 4 bytes of words and 247 stages x 16 experts x 2 bytes of
    stage counts, beyond the 15,736 bytes that W_g's padded rows (8 x 1,600), eight 24 KB stages
    and 17 barriers leave below the kernel's 220 KB."""
    chunk = -(-T_LARGE // 152)
    fixed = 8 * (768 * 2 + 64) + 8 * 16 * 768 * 2 + 17 * 8
    words = chunk * 4 + -(-chunk // 16) * 16 * 2
    assert chunk == 3948 and fixed + words > 220 * 1024


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
