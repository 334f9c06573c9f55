"""GPU parity of the CUDA layer against the CPU oracle, through the C ABI (needs a GB300).

Covers: the fp32 DeiT-T layer in full; the bf16 DeiT-S layer in full; the bf16 DeiT-B layer at
full size (routing on every token, outputs on 4,096 sampled rows plus the whole smallest expert);
the Zipf expert-count x rank sweep at its extremes; ragged, tiny, single-expert, empty-expert and
exact-tie cases; the dense FFN; run-to-run determinism and token-split invariance.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

from gpu_util import (Handle, check_routing, get_routing, handle_for, oracle_rows, out_error,
                      run_ffn, sample_rows, tol)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _full_check(L, T=None):
    s = L["shape"]
    T = T or s.T
    D = synth.to_torch(L)
    with handle_for(L, T) as h:
        out = run_ffn(h, D, T)
        gr = get_routing(h, T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    x = L["x"][:T]
    check_routing(gr, x, L["Wg"], L["bg"])
    y = oracle_rows(L, np.arange(T), gr["a"])
    err = out_error(out, y, s.dtype)
    assert err <= tol(s.dtype), f"{s.name} T={T}: error {err:.3e}"
    return err, gr


def test_deit_tiny_fp32_full(workload):
    _full_check(workload(synth.DEIT_TINY_FP32))


def test_deit_small_bf16_full(workload):
    _full_check(workload(synth.DEIT_SMALL_BF16))


@pytest.mark.parametrize("T", [1, 7, 129, 1000])
def test_ragged_token_counts(workload, T):
    _full_check(workload(synth.DEIT_SMALL_BF16), T=T)


@pytest.mark.parametrize("T", [1, 33, 300])
def test_ragged_token_counts_fp32(workload, T):
    _full_check(workload(synth.DEIT_TINY_FP32), T=T)


def test_deit_base_bf16_sampled(workload):
    L = workload(synth.DEIT_BASE_BF16)
    s = L["shape"]
    D = synth.to_torch(L)
    with handle_for(L) as h:
        out = run_ffn(h, D)
        gr = get_routing(h, s.T, s.E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    rows = sample_rows(gr, s.T)
    y = oracle_rows(L, rows, gr["a"][rows])
    err = out_error(out[torch.from_numpy(rows).cuda()], y, "bf16")
    assert err <= tol("bf16"), f"error {err:.3e}"


@pytest.mark.parametrize("E,r", [(2, 16), (2, 256), (3, 64), (8, 16), (8, 256), (6, 128)])
def test_zipf_sweep_points(E, r):
    L = synth.make_layer(synth.deit_small_zipf(E, r).with_(n_cal=4000))
    _full_check(L)


def test_single_expert_is_dense_order(workload):
    """E = 1: the permutation is the identity and every token takes expert 0."""
    L = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=777, E=1, n_cal=2000))
    _, gr = _full_check(L)
    assert np.array_equal(gr["perm"], np.arange(777))


def test_empty_and_dominant_experts():
    """A router that never picks some experts and sends most tokens to one."""
    L = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=1500, E=6, n_cal=3000))
    bg = L["bg"].copy()
    bg[[1, 4]] = -1e4           # experts 1 and 4 never win
    bg[2] += 200.0              # expert 2 wins most tokens
    L = dict(L, bg=synth.round_bf16(bg))
    _, gr = _full_check(L)
    assert gr["counts"][1] == 0 and gr["counts"][4] == 0
    assert gr["counts"][2] == gr["counts"].max() and gr["counts"][2] >= 500


def test_exact_ties_take_lowest_index():
    """Integer-valued tokens and router rows make every logit exact in fp32; duplicated rows tie
    and the lower expert index must win, bit-exactly, on the GPU."""
    rng = np.random.default_rng(11)
    L = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=600, E=4, n_cal=2000))
    x = rng.integers(-3, 4, (600, 384)).astype(np.float32)
    Wg = rng.integers(-2, 3, (4, 384)).astype(np.float32)
    Wg[3] = Wg[1]
    Wg[2] = Wg[0]
    L = dict(L, x=x, Wg=Wg, bg=np.zeros(4, np.float32))
    D = synth.to_torch(L)
    with handle_for(L) as h:
        cm.clearmoe_route(h.h, D["x"], D["Wg"], D["bg"])
        gr = get_routing(h, 600, 4)
    want = O.sort_by_expert(O.argmax_lowest(O.router_logits(x, Wg, np.zeros(4))), 4)
    assert np.array_equal(gr["a"], want["a"]) and set(gr["a"].tolist()) <= {0, 1}
    assert np.array_equal(gr["perm"], want["perm"])


def test_dense_ffn(workload):
    for shape in (synth.DEIT_TINY_FP32, synth.DEIT_SMALL_BF16):
        L = workload(shape)
        D = synth.to_torch(L)
        T = 2000 if shape.T > 2000 else shape.T
        with handle_for(L) as h:
            out = torch.empty(T, shape.d, device="cuda", dtype=D["x"].dtype)
            cm.clearmoe_dense_ffn_forward(h.h, D["x"][:T], D["W1"], D["b1"], D["W2"], out)
            torch.cuda.synchronize()
        y = O.dense_ffn(L["x"][:T], L["W1"], L["b1"], L["W2"], z_bf16=shape.dtype == "bf16")
        err = out_error(out, y, shape.dtype)
        assert err <= tol(shape.dtype), f"{shape.name}: {err:.3e}"


def test_deterministic_and_token_split(workload):
    """Two runs are bitwise equal, and forward(T) = concat(forward(T1), forward(T2)) bitwise."""
    L = workload(synth.DEIT_SMALL_BF16)
    D = synth.to_torch(L)
    T = L["shape"].T
    with handle_for(L) as h:
        a = run_ffn(h, D).clone()
        b = run_ffn(h, D).clone()
        x1, x2 = D["x"][:5000].contiguous(), D["x"][5000:].contiguous()
        o1 = run_ffn(h, dict(D, x=x1)).clone()
        o2 = run_ffn(h, dict(D, x=x2)).clone()
        torch.cuda.synchronize()
    assert torch.equal(a, b)
    assert torch.equal(torch.cat([o1, o2]), a)
    assert T == 12608


def test_fp32_split_k_deterministic(workload):
    """The fp32 layer's SIMT GEMMs split K when their tiles alone would leave the GPU idle (DeiT-T:
    the basis factor six ways, the grouped GEMM three ways); the tile's last block adds the partial
    sums in split order. Repeated forwards on one handle (whose per-tile counters clear themselves)
    are bitwise equal, and a second handle gives the same bits; the T = 1 and T = 300 launches in
    between split differently and must not disturb the counters."""
    L = workload(synth.DEIT_TINY_FP32)
    D = synth.to_torch(L)
    with handle_for(L) as h:
        a = run_ffn(h, D).clone()
        run_ffn(h, D, T=1)
        run_ffn(h, D, T=300)
        b = run_ffn(h, D).clone()
        assert cm.clearmoe_layer_status(h.h) == 0
    with handle_for(L) as h2:
        c = run_ffn(h2, D).clone()
    torch.cuda.synchronize()
    assert torch.equal(a, b) and torch.equal(a, c)
    assert torch.isfinite(a).all()


def test_bounded_wait_reports_timeout(workload):
    """The routing kernel's producer withholds its first stage copy on purpose
    (clearmoe_debug_set_wait), so the MMA thread's bounded mbarrier wait for it runs out after
    20 ms; the producer lets its other copies land before the CTA exits. The call reports
    CLEARMOE_ETIMEOUT through the status word, and the handle computes correct results afterwards."""
    L = workload(synth.DEIT_SMALL_BF16)
    D = synth.to_torch(L)
    with handle_for(L) as h:
        cm.clearmoe_debug_set_wait(h.h, 20_000_000, 1)
        cm.clearmoe_route(h.h, D["x"], D["Wg"], D["bg"])
        assert cm.clearmoe_layer_status(h.h) == cm.ETIMEOUT
        assert cm.clearmoe_layer_status(h.h) == 0
        cm.clearmoe_debug_set_wait(h.h, 1_000_000_000, 0)
        out = run_ffn(h, D)
        gr = get_routing(h, L["shape"].T, L["shape"].E)
        assert cm.clearmoe_layer_status(h.h) == 0
    check_routing(gr, L["x"], L["Wg"], L["bg"])
    assert torch.isfinite(out.float()).all()


def test_invalid_arguments_enqueue_nothing(workload):
    L = workload(synth.DEIT_SMALL_BF16)
    D = synth.to_torch(L)
    with handle_for(L, 1000) as h:
        out = torch.zeros(1001, 384, device="cuda", dtype=torch.bfloat16)
        with pytest.raises(cm.ClearMoEError) as e:  # T above max_tokens
            cm.clearmoe_ffn_forward(h.h, D["x"][:1001], D["W1"], D["b1"], D["U"], D["S"],
                                    D["Vh"], D["residuals"], D["Wg"], D["bg"], out)
        assert e.value.code == cm.EINVAL
        with pytest.raises(cm.ClearMoEError) as e:  # r not a multiple of 16 on the bf16 path
            cm.clearmoe_ffn_forward(h.h, D["x"][:100], D["W1"], D["b1"], D["U"][:, :24].contiguous(),
                                    D["S"][:24].contiguous(), D["Vh"][:24].contiguous(),
                                    D["residuals"], D["Wg"], D["bg"], out[:100])
        assert e.value.code == cm.EUNSUPPORTED
        torch.cuda.synchronize()
        assert torch.count_nonzero(out) == 0
        with pytest.raises(cm.ClearMoEError):  # routing read before any forward
            cm.clearmoe_get_routing(h.h, idx=torch.empty(10, dtype=torch.int32, device="cuda"))
