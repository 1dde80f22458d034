"""Pins of the oracle's training-step pieces (Algorithm 1 on a fully
connected layer): the fp32 AQE forward against the fp64 definition and its
alpha limits, the fp32 backward against the fp64 one, the update's single
rounding against exact rational arithmetic, and the two products of the
backward pass against finite differences of the forward product."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import oracle as O
from paper_2003_04296_gb300.inputs import DEFAULT_THR


def _x(n=4000, seed=0):
    r = np.random.default_rng(seed)
    return np.concatenate([r.standard_normal(n) * 1.3, [0.0, 1.0, -1.0, 0.5, 0.125, -0.375]]).astype(np.float32)


@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("alpha", [0.0, 0.3, 0.75, 1.0])
def test_aqe_forward_f32(bits, alpha):
    """Within two fp32 roundings of Eq. activation's value; alpha = 1 gives h,
    alpha = 0 the identity, exactly."""
    x = _x(seed=bits)
    y = O.aqe_forward_f32(x, alpha, bits, DEFAULT_THR[bits]).astype(np.float64)
    ref = O.aqe_forward(x, float(np.float32(alpha)), bits, DEFAULT_THR[bits])
    np.testing.assert_allclose(y, ref, rtol=2.0 ** -22, atol=2.0 ** -40)
    if alpha == 1.0:
        assert np.array_equal(y, O.quantize(x[None], bits, DEFAULT_THR[bits])[0])
    if alpha == 0.0:
        assert np.array_equal(y, x.astype(np.float64))


@pytest.mark.parametrize("alpha", [0.25, 0.6, 1.0])
def test_aqe_backward_f32(alpha):
    """g (2 alpha) is one exact doubling and one rounding: the fp64 value rounded."""
    x, g = _x(seed=5), _x(seed=6)
    got = O.aqe_backward_f32(x, g, alpha)
    want = O.aqe_backward(x, g, float(np.float32(alpha))).astype(np.float32)
    assert np.array_equal(got, want)


def test_sgd_clip_single_rounding():
    """min(1, max(-1, w - lr g)) with one rounding: within half an fp32 ulp of
    the exact rational value, then clipped."""
    r = np.random.default_rng(9)
    w = r.uniform(-1, 1, 300).astype(np.float32)
    g = (r.standard_normal(300) * 10.0 ** r.integers(-4, 3, 300)).astype(np.float32)
    lr = np.float32(0.01)
    got = O.sgd_clip(w, g, lr)
    for wi, gi, yi in zip(w, g, got):
        exact = Fraction(float(wi)) - Fraction(float(lr)) * Fraction(float(gi))
        if exact >= 1:
            assert yi == 1.0
        elif exact <= -1:
            assert yi == -1.0
        else:
            ulp = np.spacing(np.float32(abs(yi)))
            assert abs(Fraction(float(yi)) - exact) <= Fraction(float(ulp)) / 2


def test_backward_products_are_the_gradients():
    """For the bilinear forward a~ = A W^T, the products g_A = G W and
    g_W = G^T A (Algorithm 1's backward) are the gradients of sum(G * a~):
    central differences in fp64."""
    r = np.random.default_rng(3)
    A, W, G = r.standard_normal((4, 6)), r.standard_normal((5, 6)), r.standard_normal((4, 5))
    f = lambda A_, W_: np.sum(G * (A_ @ W_.T))
    gA, gW = G @ W, G.T @ A
    h = 1e-6
    for (i, j) in [(0, 0), (2, 3), (3, 5)]:
        E = np.zeros_like(A); E[i, j] = h
        assert abs((f(A + E, W) - f(A - E, W)) / (2 * h) - gA[i, j]) < 1e-6
    for (i, j) in [(0, 1), (4, 5), (2, 2)]:
        E = np.zeros_like(W); E[i, j] = h
        assert abs((f(A, W + E) - f(A, W - E)) / (2 * h) - gW[i, j]) < 1e-6
