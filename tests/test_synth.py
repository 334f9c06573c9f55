"""Checks of the seeded workload generator's offline conversion (no GPU).

The generator runs the paper's Phase 3 (truncated SVD, k-means, scales, residuals); these pin it
to the mathematics: orthonormal singular vectors, the Eckart-Young error of the truncation, the
monotone reconstruction error in r (the trend of the paper's rank sweep), and the identity
sum_e |C_e| s_e = N that follows from the definition of s_e in Algorithm 2.
"""
import numpy as np
import pytest

import synth


def test_svd_orthonormal_and_eckart_young():
    rng = np.random.default_rng(0)
    W2 = synth.WEIGHT_STD * rng.standard_normal((96, 384))
    for r in (8, 32, 96):
        U, S, Vh, S_all = synth.truncated_svd(W2, r)
        assert np.allclose(U.T @ U, np.eye(r), atol=1e-12)
        assert np.allclose(Vh @ Vh.T, np.eye(r), atol=1e-12)
        err = np.linalg.norm(W2 - (U * S) @ Vh, "fro") ** 2
        assert err == pytest.approx(np.sum(S_all[r:] ** 2), rel=1e-9, abs=1e-20)
        j = np.abs(U).argmax(axis=0)
        assert np.all(U[j, np.arange(r)] > 0)  # sign convention


def test_recon_error_monotone_in_rank():
    rng = np.random.default_rng(1)
    W2 = rng.standard_normal((64, 256))
    errs = []
    for r in (4, 8, 16, 32, 64):
        U, S, Vh, _ = synth.truncated_svd(W2, r)
        errs.append(np.linalg.norm(W2 - (U * S) @ Vh) / np.linalg.norm(W2))
    assert all(b <= a for a, b in zip(errs, errs[1:])) and errs[-1] < 1e-12


def test_scale_identity_and_residual_direction():
    rng = np.random.default_rng(2)
    d, H, E = 16, 64, 3
    W1 = 0.2 * rng.standard_normal((H, d))
    b1 = 0.02 * rng.standard_normal(H)
    W2 = 0.2 * rng.standard_normal((d, H))
    cent = rng.standard_normal((E, d))
    x_cal, _ = synth.mixture_tokens(rng, cent, synth.cluster_sizes(600, E, "balanced"), 0.5)
    conv = synth.convert_layer(W1, b1, W2, x_cal, E, 4, rng)
    assert np.sum(conv["cal_counts"] * conv["scales"]) == pytest.approx(600, rel=1e-12)
    assert conv["cal_counts"].sum() == 600 and np.all(conv["cal_counts"] > 0)
    # residual_e = (W2 - W_shared) s_e: every expert has the same direction
    W_sh = (conv["U"] * conv["S"]) @ conv["Vh"]
    assert np.allclose(conv["D"], W2 - W_sh, atol=1e-14)


def test_cluster_sizes_laws():
    n = synth.cluster_sizes(12608, 4, "balanced")
    assert n.tolist() == [3152] * 4
    assert synth.cluster_sizes(10, 4, "balanced").tolist() == [3, 3, 2, 2]
    for E, frac0 in ((2, 0.697), (3, 0.587), (4, 0.528), (6, 0.464), (8, 0.429)):
        z = synth.cluster_sizes(12608, E, "zipf")
        assert z.sum() == 12608 and abs(z[0] / 12608 - frac0) < 2e-3
        assert np.all(np.diff(z) <= 0)


def test_round_bf16_matches_torch():
    torch = pytest.importorskip("torch")
    v = np.random.default_rng(4).standard_normal(100000).astype(np.float32) * 7
    want = torch.from_numpy(v).to(torch.bfloat16).float().numpy()
    assert np.array_equal(synth.round_bf16(v), want)


def test_router_parameter_count_of_the_paper():
    """A linear router of d x E weights plus a bias per expert over 6 converted layers has
    (384 * 4 + 4) * 6 = 9,240 parameters at DeiT-S, the count the paper gives."""
    L = synth.make_layer(synth.DEIT_TINY_FP32.with_(T=64, d=384, H=64, n_cal=512))
    assert (L["Wg"].size + L["bg"].size) * 6 == 9240


def test_layer_shapes_and_dtype(workload):
    L = workload(synth.DEIT_TINY_FP32)
    s = L["shape"]
    assert L["x"].shape == (s.T, s.d) and L["W1"].shape == (s.H, s.d)
    assert L["U"].shape == (s.d, s.r) and L["Vh"].shape == (s.r, s.H)
    assert L["residuals"].shape == (s.E, s.d, s.H) and L["Wg"].shape == (s.E, s.d)
    assert np.allclose(L["x"].mean(1), 0, atol=1e-5)
    Lb = synth.make_layer(synth.DEIT_SMALL_BF16.with_(T=256, n_cal=1024))
    for k in ("x", "W1", "b1", "U", "Vh", "residuals", "Wg", "bg"):
        assert np.array_equal(synth.round_bf16(Lb[k]), Lb[k]), k


@pytest.mark.parametrize("dtype,bound", [("f32", 1e-5), ("bf16", 2e-2)])
def test_residual_stream_normalises_back(dtype, bound):
    """y_t = s_t x_t + m_t per token: its LayerNorm is x again, up to the eps and y's rounding."""
    x = synth.layer_norm(np.random.default_rng(4).standard_normal((128, 192)))
    y = synth.residual_stream(x, dtype)
    assert y.dtype == np.float32 and np.array_equal(y, synth.to_dtype(y, dtype))
    assert np.abs(synth.layer_norm(y) - x).max() < bound
    assert np.abs(y.mean(axis=1)).max() > 0.5  # the rows are shifted and scaled
