"""Canary-padded outputs: no entry point writes past the T rows (or T indices) it was given.

Every output buffer here has 64 extra rows (entries) after the T it is called with, filled with a
sentinel; after the call the first T rows must be finite and the tail must still hold the sentinel,
bit for bit. Covered: the forward in its forms (factorised, folded, materialised, one residual
matrix, the folded input LayerNorm, class tokens with b2, the router inside fc1 on the factorised
and folded forms), the dense FFN, the LayerNorm and the routing copies, at T = 1, 17 and 300 on the
bf16 DeiT-S layer and at T = 17 on the fp32 DeiT-T layer."""
import numpy as np
import pytest
import torch

import synth
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import handle_for

pytestmark = pytest.mark.gpu
PAD = 64
SENTINEL = 12352.0  # exact in bf16 and fp32


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _padded(T, d, dtype):
    return torch.full((T + PAD, d), SENTINEL, device="cuda", dtype=dtype)


def _check(buf, T, what):
    torch.cuda.synchronize()
    head, tail = buf[:T].float(), buf[T:].float()
    assert torch.isfinite(head).all(), f"{what}: non-finite rows below T"
    assert torch.equal(tail, torch.full_like(tail, SENTINEL)), f"{what}: wrote past row T"


@pytest.mark.parametrize("shape,T", [(synth.DEIT_SMALL_BF16, 1), (synth.DEIT_SMALL_BF16, 17),
                                     (synth.DEIT_SMALL_BF16, 300), (synth.DEIT_TINY_FP32, 17)],
                         ids=lambda v: getattr(v, "name", v))
def test_outputs_stay_within_T(workload, shape, T):
    L = workload(shape)
    D = synth.to_torch(L)
    dt = D["x"].dtype
    x = D["x"][:T]
    args = (D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"], D["Wg"], D["bg"])
    with handle_for(L) as h:
        calls = {
            "forward": lambda o: cm.clearmoe_ffn_forward(h.h, x, *args, o),
            "class tokens + b2": lambda o: cm.clearmoe_ffn_forward_ex(h.h, x, *args, o, b2=D["b2"], W2=D["W2"],
                                                                      cls_stride=197),
            "folded LayerNorm": lambda o: cm.clearmoe_ffn_forward_ex(h.h, x, *args, o, input_layernorm=True),
            "dense": lambda o: cm.clearmoe_dense_ffn_forward(h.h, x, D["W1"], D["b1"], D["W2"], o),
            "layer norm": lambda o: cm.clearmoe_layer_norm(h.h, x, o),
        }
        if shape.dtype == "bf16":
            comb = torch.empty_like(D["residuals"])
            cm.clearmoe_fold_basis(h.h, D["U"], D["S"], D["Vh"], D["residuals"], comb)
            W_sh = torch.empty(shape.d, shape.H, device="cuda", dtype=dt)
            cm.clearmoe_materialize_basis(h.h, D["U"], D["S"], D["Vh"], W_sh)
            calls["folded"] = lambda o: cm.clearmoe_ffn_forward_folded(h.h, x, D["W1"], D["b1"], comb, D["Wg"],
                                                                       D["bg"], o)
            calls["materialized"] = lambda o: cm.clearmoe_ffn_forward_materialized(
                h.h, x, D["W1"], D["b1"], W_sh, D["residuals"], D["Wg"], D["bg"], o)
            calls["scaled"] = lambda o: cm.clearmoe_ffn_forward_scaled(h.h, x, D["W1"], D["b1"], D["U"], D["S"],
                                                                       D["Vh"], D["R"], D["scales"], D["Wg"],
                                                                       D["bg"], o)
            calls["router in fc1"] = lambda o: cm.clearmoe_ffn_forward_ex(h.h, x, *args, o, router_in_fc1=True)
            calls["router in fc1, folded"] = lambda o: cm.clearmoe_ffn_forward_folded_ex(
                h.h, x, D["W1"], D["b1"], comb, D["Wg"], D["bg"], o, router_in_fc1=True)
        for what, call in calls.items():
            buf = _padded(T, shape.d, dt)
            call(buf[:T])
            _check(buf, T, what)
        routing = []  # the routing copies after the default forward and after the router inside fc1
        for fused in ((False, True) if shape.dtype == "bf16" else (False,)):
            cm.clearmoe_ffn_forward_ex(h.h, x, *args, _padded(T, shape.d, dt)[:T], router_in_fc1=fused)
            idx, perm = (torch.full((T + PAD,), -7, dtype=torch.int32, device="cuda") for _ in range(2))
            counts = torch.full((shape.E + PAD,), -7, dtype=torch.int32, device="cuda")
            offsets = torch.full((shape.E + 1 + PAD,), -7, dtype=torch.int32, device="cuda")
            cm.clearmoe_get_routing(h.h, idx, counts, offsets, perm)
            torch.cuda.synchronize()
            assert cm.clearmoe_layer_status(h.h) == 0
            routing.append((fused, idx, perm, counts, offsets))
    for fused, idx, perm, counts, offsets in routing:
        for buf, n, what in ((idx, T, "idx"), (perm, T, "perm"), (counts, shape.E, "counts"),
                             (offsets, shape.E + 1, "offsets")):
            b = buf.cpu().numpy()
            assert np.all(b[:n] >= 0) and np.all(b[n:] == -7), f"{what} (router in fc1: {fused}): wrote past its {n} entries"
