"""The bf16 layer evaluates GELU with the erf approximation of Abramowitz & Stegun 7.1.28
(Hastings): erf(x) = 1 - (1 + a1 x + ... + a6 x^6)^-16, |error| <= 3e-7. The kernel writes
GELU(u) = max(u, 0) + m y with m = -|u| / 2 and y = P^-16, running Horner's rule on m with the
coefficients (which carry 1/sqrt(2)^k) scaled by 2^k and alternating in sign, which gives -P. This
checks, on the CPU with float32 arithmetic in the kernel's order (each fma rounded once from a
float64 value, where the product is exact), that this form equals plain Horner in |u| bit for bit,
that the resulting GELU stays within 7.5e-7 of the float64 exact-erf GELU for every u, and that the
bf16-rounded hidden state it produces differs from the exactly rounded one for a negligible share
of realistic pre-activations (the rounding of z to bf16 is the layer's declared quantisation
point)."""
import numpy as np
from scipy.special import erfc

A = (0.0705230784, 0.0422820123, 0.0092705272, 0.0001520143, 0.0002765672, 0.0000430638)


def _fma32(a, b, c):
    return (a.astype(np.float64) * b.astype(np.float64) + np.asarray(c, np.float64)).astype(np.float32)


def _b():
    """b_0 .. b_6 of P(|u|) = sum b_k |u|^k, in float32."""
    return [np.float32(1)] + [np.float32(A[i] * (1 / np.sqrt(2.0)) ** (i + 1)) for i in range(6)]


def _poly_plain(au):
    b = _b()
    p = np.full_like(au, b[6])
    for k in (5, 4, 3, 2, 1, 0):
        p = _fma32(p, au, b[k])
    return p


def _poly_kernel(m):
    """The kernel's form: Horner on m = -|u| / 2 with c_k = (-1)^(k+1) b_k 2^k; returns -P."""
    c = [np.float32((-1) ** (k + 1) * float(bk) * 2.0 ** k) for k, bk in enumerate(_b())]
    p = _fma32(np.full_like(m, c[6]), m, c[5])
    for k in (4, 3, 2, 1, 0):
        p = _fma32(p, m, c[k])
    return p


def gelu_as_f32(u):
    f32 = np.float32
    u = np.asarray(u, np.float32)
    m = (f32(-0.5) * np.abs(u)).astype(f32)
    p = _poly_kernel(m)
    for _ in range(4):
        p = (p * p).astype(f32)
    with np.errstate(over="ignore", divide="ignore"):
        y = (f32(1) / p).astype(f32)
    return _fma32(m, y, np.maximum(u, f32(0)))


def gelu_exact(u):
    u = np.asarray(u, np.float64)
    return u * 0.5 * erfc(-u / np.sqrt(2.0))


def test_absolute_error_bound():
    u = np.linspace(-16, 16, 2_000_001)
    err = np.abs(gelu_as_f32(u).astype(np.float64) - gelu_exact(u.astype(np.float32)))
    assert err.max() <= 7.5e-7


def test_kernel_horner_form_is_exact():
    au = np.abs(np.random.default_rng(3).standard_normal(1_000_000).astype(np.float32) * 4)
    m = (np.float32(-0.5) * au).astype(np.float32)
    assert np.array_equal(_poly_kernel(m), -_poly_plain(au))


def test_relu_as_half_sum_is_exact():
    """The kernel forms max(u, 0) as the fma u * 0.5 + |u| / 2 (m = -|u| / 2 negated): exact
    wherever halving is (|u| >= 2^-125; below that GELU(u) rounds to zero in bf16 anyway)."""
    rng = np.random.default_rng(5)
    u = np.concatenate([rng.standard_normal(500_000) * 10.0 ** rng.integers(-30, 30, 500_000),
                        [0.0, -0.0, 2.0 ** -125, -(2.0 ** -125), 3.4e38, -3.4e38]]).astype(np.float32)
    m = (np.float32(-0.5) * np.abs(u)).astype(np.float32)
    r = _fma32(np.full_like(u, 0.5), u, -m)
    assert np.array_equal(r + np.float32(0), np.maximum(u, np.float32(0)) + np.float32(0))


def test_bf16_rounding_agrees_on_realistic_preactivations():
    torch = __import__("pytest").importorskip("torch")
    u = (np.random.default_rng(0).standard_normal(2_000_000) * 0.6).astype(np.float32)
    bf = lambda v: torch.from_numpy(np.asarray(v, np.float32)).to(torch.bfloat16).float().numpy()
    assert np.mean(bf(gelu_as_f32(u)) != bf(gelu_exact(u))) < 1e-4
