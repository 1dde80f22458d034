"""Pins of the oracle's layer pieces around the convolution (Sec. III-E:
pooling, batch normalisation, HardTanh; the fp32 first layer) against exact
rational arithmetic, textbook routines and floating-point error bounds."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import oracle as O


def round_f32(q: Fraction) -> np.float32:
    """Round an exact rational to the nearest fp32, ties to even."""
    c = np.float32(float(q))
    cands = [np.nextafter(c, np.float32(-np.inf)), c, np.nextafter(c, np.float32(np.inf))]
    best = min(cands, key=lambda v: (abs(Fraction(float(v)) - q),
                                     int(np.float32(v).view(np.uint32)) & 1))
    return np.float32(best)


def test_affine_is_single_rounding():
    """BN at inference, y = acc * scale + shift, rounded once to fp32."""
    r = np.random.default_rng(0)
    acc = r.integers(-70000, 70000, (3, 4, 5)).astype(np.int32)
    scale = r.normal(0, 0.05, 4).astype(np.float32)
    shift = r.normal(0, 0.1, 4).astype(np.float32)
    y = O.affine(acc, scale, shift)
    for b in range(3):
        for c in range(4):
            for i in range(5):
                q = Fraction(int(acc[b, c, i])) * Fraction(float(scale[c])) + Fraction(float(shift[c]))
                assert y[b, c, i] == round_f32(q)


def test_hardtanh():
    v = np.array([-3.0, -1.0, -0.5, 0.0, 0.99, 1.0, 7.0], dtype=np.float32)
    assert np.array_equal(O.hardtanh(v), np.array([-1, -1, -0.5, 0, 0.99, 1, 1], dtype=np.float32))


def test_maxpool_i32_vs_reshape():
    a = np.random.default_rng(1).integers(-100, 100, (2, 3, 6, 8)).astype(np.int32)
    ref = a.reshape(2, 3, 3, 2, 4, 2).max(axis=(3, 5))
    assert np.array_equal(O.maxpool_i32(a, 2, 2), ref)


def test_maxpool_f32_vs_torch():
    torch = pytest.importorskip("torch")
    x = np.random.default_rng(2).standard_normal((2, 3, 11, 10)).astype(np.float32)
    ref = torch.nn.functional.max_pool2d(torch.from_numpy(x), 3, 2, 1).numpy()
    assert np.array_equal(O.maxpool_f32(x, 3, 2, 1), ref)


def test_conv_f32_seq_order_and_bound():
    """The fp32 first-layer convolution is one fmaf chain over (ci, ky, kx):
    equal to an exact-rational emulation of that chain, and within the
    standard summation bound n*u*sum|x w| of the fp64 convolution."""
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(3)
    x = r.uniform(-1, 1, (1, 3, 5, 4)).astype(np.float32)
    w = np.where(r.random((2, 3, 3, 3)) < 0.5, -1.0, 1.0).astype(np.float32)
    out = O.conv2d_f32_seq(x, w, 1, 1)
    for o in range(2):
        for y in range(5):
            for xx in range(4):
                s = np.float32(0.0)
                for c in range(3):
                    for ky in range(3):
                        for kx in range(3):
                            yi, xi = y - 1 + ky, xx - 1 + kx
                            if 0 <= yi < 5 and 0 <= xi < 4:
                                s = round_f32(Fraction(float(x[0, c, yi, xi])) * Fraction(float(w[o, c, ky, kx]))
                                              + Fraction(float(s)))
                assert out[0, o, y, xx] == s
    ref = torch.nn.functional.conv2d(torch.from_numpy(x).double(), torch.from_numpy(w).double(),
                                     padding=1).numpy()
    absref = torch.nn.functional.conv2d(torch.from_numpy(np.abs(x)).double(),
                                        torch.from_numpy(np.abs(w)).double(), padding=1).numpy()
    n = 27
    u = 2.0 ** -24
    assert np.all(np.abs(out - ref) <= n * u / (1 - n * u) * absref + 1e-30)


def test_avgpool_and_linear_bounds():
    r = np.random.default_rng(4)
    x = r.standard_normal((2, 5, 7, 7)).astype(np.float32)
    avg = O.avgpool_f32(x)
    ref = x.astype(np.float64).mean(axis=(2, 3))
    assert np.all(np.abs(avg - ref) <= 60 * 2.0 ** -24 * np.abs(x).astype(np.float64).mean(axis=(2, 3)) + 1e-7)
    xf = r.standard_normal((3, 40)).astype(np.float32)
    wf = r.standard_normal((6, 40)).astype(np.float32)
    bf = r.standard_normal(6).astype(np.float32)
    y = O.linear_f32_seq(xf, wf, bf)
    ref = xf.astype(np.float64) @ wf.astype(np.float64).T + bf
    bound = 42 * 2.0 ** -24 * (np.abs(xf).astype(np.float64) @ np.abs(wf).astype(np.float64).T + np.abs(bf))
    assert np.all(np.abs(y - ref) <= bound)


def test_linear_and_avgpool_order():
    """The head's fixed operation order, which the GPU head reproduces bit for
    bit: the fully connected layer is one fmaf chain over the features in
    order (each step the exact x w + s rounded once) with the bias added last
    (one rounding); the global average pool is one fp32 sum in pixel order
    (each add rounded) and one division rounded once.  Exact rational
    emulation of both."""
    r = np.random.default_rng(6)
    x = r.standard_normal((2, 9)).astype(np.float32)
    w = r.standard_normal((3, 9)).astype(np.float32)
    b = (r.standard_normal(3) * 4).astype(np.float32)
    y = O.linear_f32_seq(x, w, b)
    for i in range(2):
        for o in range(3):
            s = np.float32(0.0)
            for k in range(9):
                s = round_f32(Fraction(float(x[i, k])) * Fraction(float(w[o, k])) + Fraction(float(s)))
            assert y[i, o] == round_f32(Fraction(float(s)) + Fraction(float(b[o])))
    t = r.standard_normal((2, 3, 5, 3)).astype(np.float32)
    avg = O.avgpool_f32(t)
    for i in range(2):
        for c in range(3):
            s = np.float32(0.0)
            for v in t[i, c].ravel():
                s = round_f32(Fraction(float(s)) + Fraction(float(v)))
            assert avg[i, c] == round_f32(Fraction(float(s)) / 15)
