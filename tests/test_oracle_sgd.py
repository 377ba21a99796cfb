"""Pins for the oracle's model update (Section 2, Eq. 1, with the aggregate in
place of the batch mean; momentum 0.9 from Appendix B, read as heavy-ball
momentum v <- mu*v + g, w <- w - eta*v with each result rounded once to fp32).

Each test checks the oracle against something fixed outside its code: exact
rational arithmetic with an fp32 round-to-nearest-even written here, a
recurrence whose values are exact dyadic numbers, and PyTorch's SGD."""
from fractions import Fraction

import numpy as np
import pytest

import oracle


def f32_round(x: Fraction) -> np.float32:
    """IEEE-754 binary32 round-to-nearest-even of a nonzero rational x."""
    assert x != 0
    neg = x < 0
    a = -x if neg else x
    e = a.numerator.bit_length() - a.denominator.bit_length()   # 2^e <= a < 2^(e+1), up to 1
    if Fraction(2) ** e > a:
        e -= 1
    elif Fraction(2) ** (e + 1) <= a:
        e += 1
    quantum = Fraction(2) ** (max(e, -126) - 23)                 # subnormals: 2^-149
    n, rem = divmod(a, quantum)
    if 2 * rem > quantum or (2 * rem == quantum and n % 2 == 1):
        n += 1
    val = n * quantum
    if val >= Fraction(2) ** 128:
        r = np.float32(np.inf)
    else:
        r = np.float32(float(val))                              # n < 2^25: exact in double
    return -r if neg else r


def fma_exact(a, b, c) -> np.float32:
    """a*b + c for finite fp32 a, b, c, computed exactly, then rounded once."""
    fa, fb, fc = (Fraction(float(x)) for x in (a, b, c))
    x = fa * fb + fc
    if x != 0:
        return f32_round(x)
    # an exact zero: -0 only when the product and the addend are both -0
    prod_neg = bool(np.signbit(a)) != bool(np.signbit(b))
    neg = fa * fb == 0 and fc == 0 and prod_neg and bool(np.signbit(c))
    return np.float32(-0.0) if neg else np.float32(0.0)


def sgd_exact(g, w, v, eta, mu):
    eta, mu = np.float32(eta), np.float32(mu)
    w2, v2 = w.copy(), None if v is None else v.copy()
    for c in range(g.size):
        if mu != 0:
            v2[c] = fma_exact(mu, v2[c], g[c])
            w2[c] = fma_exact(-eta, v2[c], w2[c])
        else:
            w2[c] = fma_exact(-eta, g[c], w2[c])
    return w2, v2


def spread(rng, n, lo=-6, hi=6):
    """fp32 values with random signs and decimal exponents in [lo, hi)."""
    return (rng.standard_normal(n) * 10.0 ** rng.uniform(lo, hi, n)).astype(np.float32)


def bits(x):
    return np.asarray(x, dtype=np.float32).view(np.uint32)


def test_rounding_helper_on_known_values():
    # pins the helper itself: values whose binary32 rounding is known
    assert bits(f32_round(Fraction(1, 3))) == 0x3EAAAAAB
    assert bits(f32_round(Fraction(1) + Fraction(1, 2 ** 24))) == 0x3F800000     # tie to even
    assert bits(f32_round(Fraction(1) + Fraction(3, 2 ** 24))) == 0x3F800002     # tie to even, up
    assert bits(f32_round(Fraction(1, 2 ** 149))) == 0x00000001                   # smallest subnormal
    assert bits(f32_round(Fraction(1, 2 ** 150))) == 0x00000000                   # tie to even: 0
    assert bits(f32_round(Fraction(3, 2 ** 151))) == 0x00000001
    assert np.isinf(f32_round(Fraction(2) ** 128))
    assert bits(f32_round(-Fraction(2) ** 127 * (2 - Fraction(1, 2 ** 23)))) == 0xFF7FFFFF


@pytest.mark.parametrize("mu", [0.9, 0.5, 0.0])
def test_sgd_matches_exact_rational_rounding(mu):
    rng = np.random.default_rng(7)
    n = 1500
    g, w, v = spread(rng, n), spread(rng, n), spread(rng, n)
    # cancellation: mu*v + g near zero, w - eta*v' near zero
    g[:200] = (-np.float32(mu) * v[:200]).astype(np.float32)
    w[200:400] = (np.float32(0.01) * g[200:400]).astype(np.float32)
    # subnormal range and near overflow
    g[400:500] = spread(rng, 100, -44, -38)
    v[400:500] = spread(rng, 100, -44, -38)
    w[500:550] = np.float32(3.0e38)
    g[500:550] = np.float32(-3.0e38)
    # signed zeros
    g[550:560] = np.float32(-0.0)
    v[550:555] = np.float32(-0.0)
    w[555:560] = np.float32(-0.0)
    eta = 0.01
    vin = None if mu == 0 else v
    w_o, v_o = oracle.sgd(g, w, vin, eta, mu)
    w_x, v_x = sgd_exact(g, w, vin, eta, mu)
    assert np.array_equal(bits(w_o), bits(w_x))
    if mu == 0:
        assert v_o is None
    else:
        assert np.array_equal(bits(v_o), bits(v_x))


def test_sgd_eq1_dyadic():
    # Eq. 1 without momentum: 1 - 0.25 * 0.5 = 0.875 exactly; v is left alone
    g = np.array([0.5, -2.0, 0.0], np.float32)
    w = np.array([1.0, 1.0, -3.0], np.float32)
    v = np.array([7.0, 7.0, 7.0], np.float32)
    w2, v2 = oracle.sgd(g, w, v, 0.25, 0.0)
    assert w2.tolist() == [0.875, 1.5, -3.0]
    assert v2.tolist() == [7.0, 7.0, 7.0]


def test_sgd_momentum_closed_form():
    # constant gradient 1, mu = 1/2, eta = 1/4, v0 = w0 = 0:
    #   v_t = 2 - 2^(1-t),  w_t = -(1/4) * (2t - 2 + 2^(1-t)), all exact in fp32
    T = 20
    g = np.ones(1, np.float32)
    w = np.zeros(1, np.float32)
    v = np.zeros(1, np.float32)
    for t in range(1, T + 1):
        w, v = oracle.sgd(g, w, v, 0.25, 0.5)
        assert v[0] == 2.0 - 2.0 ** (1 - t)
        assert w[0] == -0.25 * (2 * t - 2 + 2.0 ** (1 - t))


def test_sgd_special_values():
    inf, nan = np.float32(np.inf), np.float32(np.nan)
    g = np.array([inf, 1.0, nan, 0.0], np.float32)
    w = np.array([0.0, inf, 1.0, 1.0], np.float32)
    v = np.array([0.0, 0.0, 0.0, inf], np.float32)
    w2, v2 = oracle.sgd(g, w, v, 0.5, 0.9)
    assert v2[0] == inf and w2[0] == -inf          # v = inf, w = 0 - 0.5*inf
    assert v2[1] == 1.0 and w2[1] == inf
    assert np.isnan(v2[2]) and np.isnan(w2[2])
    assert v2[3] == inf and w2[3] == -inf


def test_sgd_rejects_missing_momentum_buffer():
    z = np.zeros(4, np.float32)
    with pytest.raises(ValueError):
        oracle.sgd(z, z, None, 0.1, 0.9)
    w2, v2 = oracle.sgd(z, z, None, 0.1, 0.0)
    assert v2 is None and np.array_equal(w2, z)


def test_sgd_agrees_with_torch_optimizer():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(11)
    n, lr, mom = 4096, 0.05, 0.9
    w0 = rng.standard_normal(n).astype(np.float32)
    p = torch.nn.Parameter(torch.from_numpy(w0.copy()))
    opt = torch.optim.SGD([p], lr=lr, momentum=mom)
    w, v = w0.copy(), np.zeros(n, np.float32)
    for _ in range(6):
        g = (rng.standard_normal(n) * 0.1).astype(np.float32)
        p.grad = torch.from_numpy(g.copy())
        opt.step()
        w, v = oracle.sgd(g, w, v, lr, mom)
        buf = opt.state[p]["momentum_buffer"].numpy()
        # PyTorch rounds mu*v and the sum separately; the oracle rounds once
        assert np.allclose(v, buf, rtol=4e-7, atol=1e-7)
        assert np.allclose(w, p.detach().numpy(), rtol=4e-7, atol=1e-7)
