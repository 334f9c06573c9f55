"""Seeded synthetic workloads for one CLEAR-MoE FFN layer (and a 12-sublayer stack).

The paper (arxiv 2606.28516) measures on DeiT/ViT activations of Imagenette images with
pretrained weights; neither is available here, so every tensor is drawn from a seeded recipe
with the shapes and structure of those workloads:

* tokens: a Gaussian mixture (centroids N(0, 1)^d, within-cluster sigma 0.5), cluster sizes
  balanced or Zipf(1.2), then layer-normalised per token (no affine, biased variance, eps 1e-6);
* fc1 W1 [H x d], b1 [H] and fc2 W2 [d x H] drawn i.i.d. N(0, 0.02^2).

It then runs the paper's *offline* conversion, whose outputs are inputs of the forward pass on
both sides of every parity test (Section "Phase 3: Expert Extraction", Eq. 2 and Algorithm 2,
and a closed-form stand-in for the Phase 4 router fit):

* truncated SVD of W2 (LAPACK through numpy) -> U_r [d x r], S_r [r], Vh_r [r x H];
* k-means (k = E, k-means++ seeding, Lloyd) on calibration hidden states GELU(W1 x + b1);
* s_e = (mean norm of hidden states in cluster e) / (mean norm over all), Algorithm 2;
* residual_e = (W2 - U_r diag(S_r) Vh_r) * s_e, Algorithm 2;
* a nearest-centroid linear router W_g[e] = m_e, b_g[e] = -|m_e|^2 / 2, m_e = mean calibration
  token of cluster e (the paper trains the router with cross-entropy on the k-means labels).

Nothing here is the forward pass being checked (routing, fc1, the shared basis, the residual
experts applied to the tokens): the oracle and the CUDA library each implement that on their own.
For bf16 workloads every tensor is rounded once to bf16 (round to nearest even) and held in
float32 arrays whose values are exactly representable in bf16; S_r stays float32.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np

LN_EPS = 1e-6
WEIGHT_STD = 0.02


@dataclass(frozen=True)
class LayerShape:
    """One converted FFN layer: T tokens of width d, hidden H = 4d, E experts, SVD rank r."""

    name: str
    T: int
    d: int
    H: int
    E: int
    r: int
    dtype: str  # "f32" or "bf16"
    sizes: str = "balanced"  # mixture cluster sizes: "balanced" or "zipf"
    clusters: int = 0  # mixture components (0 -> E)
    sigma: float = 0.5
    n_cal: int = 200 * 197  # calibration tokens: 200 images x 197 tokens (Phase 1)
    seed: int = 0

    @property
    def n_clusters(self) -> int:
        return self.clusters or self.E

    def with_(self, **kw) -> "LayerShape":
        return dataclasses.replace(self, **kw)


# The paper's backbones (Table "Cross-backbone generalization") at ViT token counts.
DEIT_TINY_FP32 = LayerShape("deit_tiny_fp32_T788", 788, 192, 768, 4, 32, "f32")
DEIT_SMALL_BF16 = LayerShape("deit_small_bf16_T12608", 12608, 384, 1536, 4, 64, "bf16")
DEIT_BASE_BF16 = LayerShape("deit_base_bf16_T50432", 50432, 768, 3072, 8, 128, "bf16")


def deit_small_zipf(E: int, r: int, seed: int = 0) -> LayerShape:
    """DeiT-S shape with Zipf(1.2) cluster sizes, for the expert-count x rank sweep."""
    return LayerShape(f"deit_small_zipf_E{E}_r{r}", 12608, 384, 1536, E, r, "bf16",
                      sizes="zipf", seed=seed)


ZIPF_E = (2, 3, 4, 6, 8)
ZIPF_R = (16, 32, 64, 128, 256)


@dataclass(frozen=True)
class StackShape:
    """12 sequential ViT-B FFN sublayers; odd blocks converted; x_{l+1} = LN(y_l)."""

    name: str = "vit_base_stack12_T100864"
    T: int = 100864
    d: int = 768
    H: int = 3072
    E: int = 8
    r: int = 128
    layers: int = 12
    moe_layers: tuple = (1, 3, 5, 7, 9, 11)
    n_cal: int = 16 * 197
    seed: int = 0


VIT_BASE_STACK12 = StackShape()


# ----------------------------------------------------------------------------------------
# elementary draws
# ----------------------------------------------------------------------------------------
def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round to the nearest bf16 (ties to even); returns float32 holding bf16 values."""
    f = np.array(a, dtype=np.float32, copy=True, order="C")
    u = f.reshape(-1).view(np.uint32)
    for s in range(0, u.size, 1 << 22):  # in place, in chunks (elementwise: same bits)
        v = u[s:s + (1 << 22)]
        lsb = (v >> 16) & 1
        v += np.uint32(0x7FFF)
        v += lsb
        v &= np.uint32(0xFFFF0000)
    return f


def to_dtype(a: np.ndarray, dtype: str) -> np.ndarray:
    a32 = np.asarray(a, dtype=np.float32)
    return round_bf16(a32) if dtype == "bf16" else np.ascontiguousarray(a32)


def cluster_sizes(T: int, C: int, law: str) -> np.ndarray:
    if law == "balanced":
        n = np.full(C, T // C, dtype=np.int64)
        n[: T - n.sum()] += 1
        return n
    if law == "zipf":
        p = np.arange(1, C + 1, dtype=np.float64) ** -1.2
        n = np.rint(T * p / p.sum()).astype(np.int64)
        n[0] += T - n.sum()
        return n
    raise ValueError(law)


def layer_norm(x: np.ndarray) -> np.ndarray:
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS)


def residual_stream(x: np.ndarray, dtype: str, seed: int = 7, scale=(0.5, 4.0), shift: float = 1.0):
    """An un-normalised stream y whose per-token LayerNorm is x again (x's rows have mean 0 and
    variance 1; up to the eps and the rounding of y): y_t = s_t x_t + m_t with s_t ~ U(scale) and
    m_t ~ N(0, shift^2) drawn per token, rounded to the layer dtype."""
    rng = np.random.default_rng(seed)
    T = x.shape[0]
    s = rng.uniform(scale[0], scale[1], size=(T, 1))
    m = shift * rng.standard_normal((T, 1))
    return to_dtype(np.asarray(x, np.float64) * s + m, dtype)


def mixture_tokens(rng: np.random.Generator, centroids: np.ndarray, sizes: np.ndarray,
                   sigma: float, chunk: int = 65536):
    """Tokens mu_label + sigma N(0, I), layer-normalised. Drawn in row chunks: consecutive draws
    continue the generator's stream, so the values equal one draw of the whole matrix while the
    temporaries stay small."""
    labels = rng.permutation(np.repeat(np.arange(len(sizes)), sizes))
    x = np.empty((labels.size, centroids.shape[1]), dtype=np.float64)
    for s in range(0, labels.size, chunk):
        lab = labels[s:s + chunk]
        x[s:s + chunk] = layer_norm(centroids[lab] + sigma * rng.standard_normal((lab.size, centroids.shape[1])))
    return x, labels


def _gelu32(u: np.ndarray) -> np.ndarray:
    from scipy.special import erf
    u = np.asarray(u, dtype=np.float32)
    return (0.5 * u * (1.0 + erf(u * np.float32(1.0 / np.sqrt(2.0))))).astype(np.float32)


def _hidden(x: np.ndarray, W1: np.ndarray, b1: np.ndarray, chunk: int = 8192) -> np.ndarray:
    """Calibration hidden states GELU(W1 x + b1) in float32 (only shapes the experts)."""
    out = np.empty((x.shape[0], W1.shape[0]), dtype=np.float32)
    W1t = np.ascontiguousarray(W1.T, dtype=np.float32)
    for s in range(0, x.shape[0], chunk):
        out[s:s + chunk] = _gelu32(x[s:s + chunk].astype(np.float32) @ W1t + b1)
    return out


# ----------------------------------------------------------------------------------------
# offline conversion (Algorithm 2 + router stand-in)
# ----------------------------------------------------------------------------------------
def truncated_svd(W2: np.ndarray, r: int):
    """W2 = U diag(S) Vh; keep the top r. Sign: the largest-magnitude entry of each u_i > 0."""
    U, S, Vh = np.linalg.svd(np.asarray(W2, dtype=np.float64), full_matrices=False)
    j = np.abs(U).argmax(axis=0)
    sgn = np.where(U[j, np.arange(U.shape[1])] < 0, -1.0, 1.0)
    U = U * sgn
    Vh = Vh * sgn[:, None]
    return U[:, :r], S[:r], Vh[:r], S


def kmeans(z: np.ndarray, k: int, rng: np.random.Generator, iters: int = 100, n_init: int = 3):
    """k-means++ seeding then Lloyd until no label changes (<= iters); the best of n_init
    seedings by inertia is kept. Distance ties go to the lowest centroid id. A cluster that
    empties is re-seeded with the point farthest from its own centroid."""
    z = np.asarray(z, dtype=np.float32)
    n = z.shape[0]
    zz = np.einsum("ij,ij->i", z, z, dtype=np.float64)

    def d2(c):
        cc = np.einsum("ij,ij->i", c, c, dtype=np.float64)
        g = z @ c.T.astype(np.float32)
        return np.maximum(zz[:, None] - 2.0 * g + cc[None, :], 0.0)

    best_labels, best_inertia = None, np.inf
    for _ in range(n_init):
        cent = np.empty((k, z.shape[1]), dtype=np.float64)
        cent[0] = z[rng.integers(n)]
        near = d2(cent[:1])[:, 0]
        for j in range(1, k):
            p = near / near.sum() if near.sum() > 0 else np.full(n, 1.0 / n)
            cent[j] = z[rng.choice(n, p=p)]
            near = np.minimum(near, d2(cent[j:j + 1])[:, 0])
        labels = np.full(n, -1, dtype=np.int64)
        for _ in range(iters):
            dist = d2(cent)
            new = dist.argmin(axis=1)
            for e in range(k):
                if not np.any(new == e):
                    own = dist[np.arange(n), new]
                    new[int(own.argmax())] = e
            if np.array_equal(new, labels):
                break
            labels = new
            for e in range(k):
                cent[e] = z[labels == e].mean(axis=0, dtype=np.float64)
        inertia = d2(cent)[np.arange(n), labels].sum()
        if inertia < best_inertia:
            best_labels, best_inertia = labels, inertia
    return best_labels


def convert_layer(W1, b1, W2, x_cal, E: int, r: int, rng: np.random.Generator):
    """Phase 3 (Algorithm 2) + router stand-in on calibration tokens x_cal (float64)."""
    U_r, S_r, Vh_r, S_all = truncated_svd(W2, r)
    z = _hidden(x_cal, W1, b1)
    labels = kmeans(z, E, rng)
    norms = np.sqrt(np.einsum("ij,ij->i", z, z, dtype=np.float64))
    counts = np.bincount(labels, minlength=E)
    s = np.array([norms[labels == e].mean() if counts[e] else 0.0 for e in range(E)])
    s = s / norms.mean()
    W_sh = (U_r * S_r) @ Vh_r
    D = np.asarray(W2, dtype=np.float64) - W_sh
    m = np.stack([x_cal[labels == e].mean(axis=0) if counts[e] else np.zeros(x_cal.shape[1])
                  for e in range(E)])
    Wg = m
    bg = -0.5 * np.einsum("ij,ij->i", m, m)
    return dict(U=U_r, S=S_r, Vh=Vh_r, sigma_all=S_all, D=D, scales=s, cal_labels=labels,
                cal_counts=counts, Wg=Wg, bg=bg)


# ----------------------------------------------------------------------------------------
# public entry points
# ----------------------------------------------------------------------------------------
def make_layer(shape: LayerShape) -> dict:
    """All inputs of one layer's forward (float32 arrays; bf16-exact values for bf16)."""
    rng = np.random.default_rng(shape.seed)
    C = shape.n_clusters
    centroids = rng.standard_normal((C, shape.d))
    x, labels = mixture_tokens(rng, centroids, cluster_sizes(shape.T, C, shape.sizes),
                               shape.sigma)
    W1 = WEIGHT_STD * rng.standard_normal((shape.H, shape.d))
    b1 = WEIGHT_STD * rng.standard_normal(shape.H)
    W2 = WEIGHT_STD * rng.standard_normal((shape.d, shape.H))
    dt = shape.dtype
    x, W1, b1, W2 = (to_dtype(a, dt) for a in (x, W1, b1, W2))

    crng = np.random.default_rng(shape.seed + 1)
    x_cal, _ = mixture_tokens(crng, centroids, cluster_sizes(shape.n_cal, C, "balanced"),
                              shape.sigma)
    x_cal = to_dtype(x_cal, dt).astype(np.float64)
    conv = convert_layer(W1, b1, W2, x_cal, shape.E, shape.r, crng)
    res = np.stack([to_dtype(conv["D"] * s, dt) for s in conv["scales"]])
    # fc2's bias (a pretrained ViT layer has one; Eq. 2 is printed without it), from its own stream
    b2 = to_dtype(WEIGHT_STD * np.random.default_rng(shape.seed + 2).standard_normal(shape.d), dt)
    return dict(
        shape=shape, dtype=dt, x=x, W1=W1, b1=b1, W2=W2, b2=b2, R=to_dtype(conv["D"], dt),
        U=to_dtype(conv["U"], dt), S=conv["S"].astype(np.float32), Vh=to_dtype(conv["Vh"], dt),
        residuals=res, Wg=to_dtype(conv["Wg"], dt), bg=to_dtype(conv["bg"], dt),
        scales=conv["scales"], labels=labels, sigma_all=conv["sigma_all"],
        cal_counts=conv["cal_counts"],
    )


def make_stack(shape: StackShape = VIT_BASE_STACK12, T: int | None = None) -> dict:
    """Inputs of the 12-sublayer stack. Layer l has seed 1000 + l; odd layers are CLEAR-MoE.

    Calibration tokens are pushed through the preceding sublayers with their dense fc2
    (float32) and layer-normalised, so each converted layer is calibrated on its own inputs.
    """
    T = shape.T if T is None else T
    rng = np.random.default_rng(shape.seed)
    centroids = rng.standard_normal((shape.E, shape.d))
    x, _ = mixture_tokens(rng, centroids, cluster_sizes(T, shape.E, "balanced"), 0.5)
    crng = np.random.default_rng(shape.seed + 1)
    x_cal, _ = mixture_tokens(crng, centroids, cluster_sizes(shape.n_cal, shape.E, "balanced"),
                              0.5)
    layers = []
    for l in range(shape.layers):
        lrng = np.random.default_rng(1000 + l)
        W1 = round_bf16(WEIGHT_STD * lrng.standard_normal((shape.H, shape.d)))
        b1 = round_bf16(WEIGHT_STD * lrng.standard_normal(shape.H))
        W2 = round_bf16(WEIGHT_STD * lrng.standard_normal((shape.d, shape.H)))
        xc = round_bf16(x_cal).astype(np.float64)
        L = dict(W1=W1, b1=b1, W2=W2, moe=l in shape.moe_layers)
        if L["moe"]:
            conv = convert_layer(W1, b1, W2, xc, shape.E, shape.r, lrng)
            L.update(U=round_bf16(conv["U"]), S=conv["S"].astype(np.float32),
                     Vh=round_bf16(conv["Vh"]),
                     residuals=np.stack([round_bf16(conv["D"] * s) for s in conv["scales"]]),
                     Wg=round_bf16(conv["Wg"]), bg=round_bf16(conv["bg"]),
                     scales=conv["scales"], E=shape.E, r=shape.r)
        layers.append(L)
        x_cal = layer_norm(_hidden(xc, W1, b1) @ W2.T.astype(np.float32))
    return dict(shape=shape, dtype="bf16", x=round_bf16(x), layers=layers, T=T)


def mlp_router(layer: dict, hidden: int | None = None, act: str = "relu") -> dict:
    """Weights of an MLP router d -> hidden -> E (Phase 4 "MLP", hidden = d / 6 by default) built
    from the layer's linear router, so that it routes the mixture as sensibly without training.

    P (rows) is an orthonormal basis of the span of W_g's rows; hidden units 0..E-1 read P x and
    units E..2E-1 read -P x, and since act(u) - act(-u) = u for ReLU and for GELU, output weights
    [W_g P^T, -W_g P^T] reproduce W_g P^T P x = W_g x. The remaining units get random input
    weights and small random output weights, which perturb the decisions near cluster borders.
    Values are rounded to the layer dtype like every other weight."""
    Wg = np.asarray(layer["Wg"], np.float64)
    bg = np.asarray(layer["bg"], np.float64)
    E, d = Wg.shape
    hidden = hidden or d // 6
    if hidden < 2 * E:
        raise ValueError("the MLP router needs at least 2 E hidden units")
    P = np.linalg.qr(Wg.T)[0].T  # E x d, orthonormal rows
    rng = np.random.default_rng(layer["shape"].seed + 3)
    W_in = np.zeros((hidden, d))
    W_in[:E], W_in[E:2 * E] = P, -P
    W_in[2 * E:] = rng.standard_normal((hidden - 2 * E, d)) / np.sqrt(d)
    b_in = np.zeros(hidden)
    b_in[2 * E:] = 0.1 * rng.standard_normal(hidden - 2 * E)
    G = Wg @ P.T
    W_out = np.zeros((E, hidden))
    W_out[:, :E], W_out[:, E:2 * E] = G, -G
    W_out[:, 2 * E:] = 0.05 * np.abs(G).mean() * rng.standard_normal((E, hidden - 2 * E))
    dt = layer["dtype"]
    return dict(W_in=to_dtype(W_in, dt), b_in=to_dtype(b_in, dt), W_out=to_dtype(W_out, dt),
                b_out=to_dtype(bg, dt), hidden=hidden, act=act)


def to_torch(layer: dict, device="cuda") -> dict:
    """Device copies of a layer's arrays in its dtype (bf16 values convert exactly); S_r and
    the integer metadata keep their types."""
    import torch

    tdt = torch.bfloat16 if layer.get("dtype", "bf16") == "bf16" else torch.float32
    out = {}
    for k in ("x", "W1", "b1", "W2", "b2", "R", "U", "Vh", "residuals", "Wg", "bg", "W_in", "b_in", "W_out",
              "b_out"):
        if k in layer:
            out[k] = torch.from_numpy(np.ascontiguousarray(layer[k], dtype=np.float32)).to(
                device=device, dtype=tdt).contiguous()
    for k in ("S", "scales"):  # fp32 in every layer dtype
        if k in layer:
            out[k] = torch.from_numpy(np.ascontiguousarray(layer[k], dtype=np.float32)).to(device)
    return out
