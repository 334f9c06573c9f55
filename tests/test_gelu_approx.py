"""The bf16 layer evaluates GELU with the erf approximation of Abramowitz & Stegun 7.1.28
(Hastings): erf(x) = 1 - (1 + a1 x + ... + a6 x^6)^-16, |error| <= 3e-7. This checks, on the CPU
with float32 arithmetic in the kernel's order, that the resulting GELU stays within 7.5e-7 of the
float64 exact-erf GELU for every u, and that the bf16-rounded hidden state it produces differs from
the exactly rounded one for a negligible share of realistic pre-activations (the rounding of z to
bf16 is the layer's declared quantisation point)."""
import numpy as np
from scipy.special import erfc

A = (0.0705230784, 0.0422820123, 0.0092705272, 0.0001520143, 0.0002765672, 0.0000430638)


def gelu_as_f32(u):
    f32 = np.float32
    b = [f32(A[i] * (1 / np.sqrt(2.0)) ** (i + 1)) for i in range(6)]
    u = np.asarray(u, np.float32)
    au = np.abs(u)
    p = b[5]
    for c in (b[4], b[3], b[2], b[1], b[0], f32(1)):
        p = (p * au + c).astype(f32)
    for _ in range(4):
        p = (p * p).astype(f32)
    with np.errstate(over="ignore", divide="ignore"):
        y = (f32(1) / p).astype(f32)
    h = (f32(0.5) * u * y).astype(f32)
    return np.where(u >= 0, u - h, h)


def gelu_exact(u):
    u = np.asarray(u, np.float64)
    return u * 0.5 * erfc(-u / np.sqrt(2.0))


def test_absolute_error_bound():
    u = np.linspace(-16, 16, 2_000_001)
    err = np.abs(gelu_as_f32(u).astype(np.float64) - gelu_exact(u.astype(np.float32)))
    assert err.max() <= 7.5e-7


def test_bf16_rounding_agrees_on_realistic_preactivations():
    torch = __import__("pytest").importorskip("torch")
    u = (np.random.default_rng(0).standard_normal(2_000_000) * 0.6).astype(np.float32)
    bf = lambda v: torch.from_numpy(np.asarray(v, np.float32)).to(torch.bfloat16).float().numpy()
    assert np.mean(bf(gelu_as_f32(u)) != bf(gelu_exact(u))) < 1e-4
