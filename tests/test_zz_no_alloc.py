"""clearmoe_route_noalloc, the routing entry point for callers that cannot allocate device memory
(engines that own every device byte, fixed memory budgets, loops that cannot afford cudaMalloc's
device synchronisation): it keeps its scratch in a static device array instead of a handle's
workspace. Checked through the C ABI against clearmoe_route, bit-exactly, on two calls in a row
that reuse the same scratch (the second with a different token count and expert count), on the fp32
routing kernel with and without a status word; tests/test_gpu_large_tokens.py runs it at 600,000
tokens, where the per-row words live in the caller's idx between the two kernels.
This file is collected last on purpose, so a failure here leaves every other test already run."""
import numpy as np
import pytest
import torch

import synth
from paper_2606_28516_gb300 import clearmoe as cm

pytestmark = pytest.mark.gpu


def _handle_routing(L, T):
    s = L["shape"]
    D = synth.to_torch(L)
    h = cm.clearmoe_layer_create(T, s.d, s.H, s.E, s.r, cm.BF16 if s.dtype == "bf16" else cm.F32)
    try:
        x = D["x"][:T].contiguous()
        cm.clearmoe_route(h, x, D["Wg"], D["bg"])
        out = [torch.empty(n, dtype=torch.int32, device="cuda") for n in (T, s.E, s.E + 1, T)]
        cm.clearmoe_get_routing(h, *out)
        torch.cuda.synchronize()
        assert cm.clearmoe_layer_status(h) == 0
    finally:
        cm.clearmoe_layer_destroy(h)
    return x, D, [o.cpu().numpy() for o in out]


def test_route_noalloc_matches_route_twice():
    import __graft_entry__
    __graft_entry__.build()
    cases = [synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=3000, n_cal=2000)),
             synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=12608, E=6, n_cal=2000, seed=3))]
    for L in cases:
        s = L["shape"]
        x, D, want = _handle_routing(L, s.T)
        got = [torch.full((n,), -7, dtype=torch.int32, device="cuda") for n in (s.T, s.E, s.E + 1, s.T)]
        status = torch.full((1,), -7, dtype=torch.int32, device="cuda")
        cm.clearmoe_route_noalloc(x, D["Wg"], D["bg"], *got, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        for g, w, name in zip(got, want, ("idx", "counts", "offsets", "perm")):
            assert np.array_equal(g.cpu().numpy(), w), name


def test_route_noalloc_fp32_and_without_status_word():
    """The fp32 routing kernel (two CTAs per SM, one token per lane) through the same entry point,
    once with a status word and once without one (the array's spare word takes the status then),
    bit for bit against the handle's routing."""
    import __graft_entry__
    __graft_entry__.build()
    L = synth.make_layer(synth.DEIT_TINY_FP32)
    s = L["shape"]
    x, D, want = _handle_routing(L, s.T)
    for status in (torch.full((1,), -7, dtype=torch.int32, device="cuda"), None):
        got = [torch.full((n,), -7, dtype=torch.int32, device="cuda") for n in (s.T, s.E, s.E + 1, s.T)]
        cm.clearmoe_route_noalloc(x, D["Wg"], D["bg"], *got, status=status)
        torch.cuda.synchronize()
        if status is not None:
            assert int(status.item()) == 0
        for g, w, name in zip(got, want, ("idx", "counts", "offsets", "perm")):
            assert np.array_equal(g.cpu().numpy(), w), name


def test_route_noalloc_rejects_bad_sizes():
    L = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=64, n_cal=1000))
    D = synth.to_torch(L)
    o = [torch.empty(64, dtype=torch.int32, device="cuda") for _ in range(4)]
    Wg17 = torch.zeros(17, 384, dtype=torch.bfloat16, device="cuda")
    b17 = torch.zeros(17, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(cm.ClearMoEError) as e:
        cm.clearmoe_route_noalloc(D["x"], Wg17, b17, *o)
    assert e.value.code == cm.EINVAL
    with pytest.raises(cm.ClearMoEError) as e:
        cm.clearmoe_route_noalloc(D["x"][:, :96].contiguous(), D["Wg"][:, :96].contiguous(), D["bg"], *o)
    assert e.value.code == cm.EUNSUPPORTED
