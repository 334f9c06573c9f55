"""Helpers of the GPU parity tests: run the library through its C ABI, compare with the oracle.

Comparison rules (the layer's stated tolerances):
  * routing: expert index bit-exact except tokens whose top-2 router logits differ by less than
    1e-5 relative (the oracle flags them); counts must equal the histogram of the GPU's indices,
    and the permutation must be exactly the stable sort of the GPU's indices;
  * fp32 layer: ||out - y||_2 / ||y||_2 <= 1e-4 against the float64 oracle;
  * bf16 layer: max |out - y| / RMS(y) <= 2e-2 against the oracle with its hidden state z stored
    in bf16 (the layer's declared quantisation point); the oracle follows the GPU's expert choice
    only on flagged near-tie tokens.
"""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import clearmoe as O
from paper_2606_28516_gb300 import clearmoe as cm

TOL_F32_REL_L2 = 1e-4
TOL_BF16_MAX_OVER_RMS = 2e-2


class Handle:
    def __init__(self, T, d, H, E, r, dtype):
        self.h = cm.clearmoe_layer_create(T, d, H, E, r, cm.BF16 if dtype == "bf16" else cm.F32)

    def close(self):
        if self.h:
            cm.clearmoe_layer_destroy(self.h)
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()


def handle_for(L: dict, max_tokens=None) -> Handle:
    s = L["shape"]
    return Handle(max_tokens or s.T, s.d, s.H, s.E, s.r, s.dtype)


def run_ffn(h: Handle, D: dict, T=None):
    x = D["x"] if T is None else D["x"][:T]
    out = torch.full((x.shape[0], D["W1"].shape[1]), float("nan"), device="cuda", dtype=x.dtype)
    cm.clearmoe_ffn_forward(h.h, x, D["W1"], D["b1"], D["U"], D["S"], D["Vh"], D["residuals"],
                            D["Wg"], D["bg"], out)
    return out


def get_routing(h: Handle, T: int, E: int):
    idx = torch.empty(T, dtype=torch.int32, device="cuda")
    perm = torch.empty(T, dtype=torch.int32, device="cuda")
    counts = torch.empty(E, dtype=torch.int32, device="cuda")
    offsets = torch.empty(E + 1, dtype=torch.int32, device="cuda")
    cm.clearmoe_get_routing(h.h, idx=idx, counts=counts, offsets=offsets, perm=perm)
    torch.cuda.synchronize()
    return dict(a=idx.cpu().numpy().astype(np.int64), counts=counts.cpu().numpy().astype(np.int64),
                offsets=offsets.cpu().numpy().astype(np.int64),
                perm=perm.cpu().numpy().astype(np.int64))


def check_routing(gpu: dict, x, Wg, bg) -> dict:
    """Asserts the routing rules; returns the oracle routing and the mismatch count."""
    E = np.asarray(Wg).shape[0]
    rt = O.route(x, Wg, bg)
    free = ~rt["near_tie"]
    bad = int(np.sum(gpu["a"][free] != rt["a"][free]))
    assert bad == 0, f"{bad} tokens routed differently (outside near ties)"
    assert np.all((gpu["a"] >= 0) & (gpu["a"] < E))
    want = O.sort_by_expert(gpu["a"], E)
    assert np.array_equal(gpu["counts"], want["counts"]), "counts != histogram of indices"
    assert np.array_equal(gpu["offsets"], want["offsets"]), "offsets != prefix sum of counts"
    assert np.array_equal(gpu["perm"], want["perm"]), "perm != stable sort by expert"
    return rt


def out_error(got: torch.Tensor, y: np.ndarray, dtype: str) -> float:
    g = got.float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(g)), "non-finite outputs"
    if dtype == "bf16":
        return float(np.abs(g - y).max() / np.sqrt(np.mean(y ** 2)))
    return float(np.linalg.norm(g - y) / np.linalg.norm(y))


def tol(dtype: str) -> float:
    return TOL_BF16_MAX_OVER_RMS if dtype == "bf16" else TOL_F32_REL_L2


def oracle_rows(L: dict, rows, a_rows):
    """Oracle output of the given token rows with the given expert choices."""
    return O.ffn_forward(L["x"][rows], L["W1"], L["b1"], L["U"], L["S"], L["Vh"],
                         L["residuals"], a=a_rows, z_bf16=L["dtype"] == "bf16")


def sample_rows(gpu_routing: dict, T: int, n: int = 4096, seed: int = 0) -> np.ndarray:
    """A seeded sample of rows plus every row of the smallest non-empty expert."""
    rng = np.random.default_rng(seed)
    rows = rng.choice(T, size=min(n, T), replace=False)
    c = gpu_routing["counts"]
    nz = np.nonzero(c)[0]
    e = nz[np.argmin(c[nz])]
    small = np.nonzero(gpu_routing["a"] == e)[0]
    return np.unique(np.concatenate([rows, small]))
