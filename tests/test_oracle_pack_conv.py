"""Pins of the oracle's bit-plane packing and of its convolution of quantized
levels (Algorithm 1 inference product) against hand-worked words, the
XNOR/popcount identities of Sec. III-C / Table I and a textbook convolution."""
import os
from itertools import product

import numpy as np
import pytest

from oracle import oracle as O
from paper_2003_04296_gb300.inputs import DEFAULT_THR

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "pack_small.txt")


def _golden():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            b, lv, words = [s.strip() for s in line.split("|")]
            rows.append((int(b), [float(v) for v in lv.split()], [int(w, 16) for w in words.split()]))
    return rows


@pytest.mark.parametrize("bits,levels,words", _golden())
def test_pack_golden(bits, levels, words):
    lv = np.array(levels, dtype=np.float64).reshape(1, -1, 1, 1)
    out = O.pack(lv, bits)
    assert out.ravel().tolist() == words


def _decode(planes, bits, C):
    """Independent decoder written from the layout description."""
    N, H, W, P, NW = planes.shape
    lv = np.zeros((N, C, H, W))
    for n, y, x, c in product(range(N), range(H), range(W), range(C)):
        bit = lambda p: (int(planes[n, y, x, p, c // 32]) >> (c % 32)) & 1
        neg = bit(0)
        if bits == 1:
            v = -1.0 if neg else 1.0
        elif bits == 2:
            v = (-1.0 if neg else 1.0) * bit(1)
        else:
            k = bit(1) | (bit(2) << 1)
            v = 0.0 if k == 0 else (-1.0 if neg else 1.0) * 2.0 ** (k - 3)
        lv[n, c, y, x] = v
    return lv


@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("C", [5, 32, 45, 64])
def test_pack_roundtrip_and_tail(bits, C):
    x = np.random.default_rng(C * 10 + bits).standard_normal((2, C, 3, 2)).astype(np.float32)
    lv = O.quantize(x, bits, DEFAULT_THR[bits])
    planes = O.pack(lv, bits)
    assert planes.shape == (2, 3, 2, bits, (C + 31) // 32)
    assert np.array_equal(_decode(planes, bits, C), lv)
    if C % 32:
        tail_mask = np.uint32((0xFFFFFFFF << (C % 32)) & 0xFFFFFFFF)
        assert not np.any(planes[..., -1] & tail_mask)
    if bits == 3:  # a zero level carries sign bit 0
        zero = lv == 0
        assert np.all(_decode(planes, 1, C)[zero] == 1.0)


def _popc(v):
    return bin(v).count("1")


@pytest.mark.parametrize("K", [1, 31, 32, 100, 4608])
def test_xnor_popcount_identity(K):
    """For +-1 vectors, dot(a, w) = K - 2 popc(a XOR w) on sign bits (the XNOR
    inference of Table I, 1-bit x 1-bit)."""
    r = np.random.default_rng(K)
    a = np.where(r.random(K) < 0.5, -1.0, 1.0)
    w = np.where(r.random(K) < 0.5, -1.0, 1.0)
    acc = O.conv2d_levels(a.reshape(1, K, 1, 1), w.reshape(1, K, 1, 1), 1, 0, 1, 1)
    sa = int("".join("1" if v < 0 else "0" for v in a), 2)
    sw = int("".join("1" if v < 0 else "0" for v in w), 2)
    assert acc.item() == K - 2 * _popc(sa ^ sw)


@pytest.mark.parametrize("K", [7, 64, 513])
def test_ternary_popcount_identity(K):
    """Ternary (2-bit) levels: dot = popc(Ma & Mw) - 2 popc(Ma & Mw & (Sa ^ Sw))."""
    r = np.random.default_rng(K)
    a = r.choice([-1.0, 0.0, 1.0], K)
    w = r.choice([-1.0, 0.0, 1.0], K)
    acc = O.conv2d_levels(a.reshape(1, K, 1, 1), w.reshape(1, K, 1, 1), 1, 0, 2, 2)
    bits = lambda cond: int("".join("1" if c else "0" for c in cond), 2)
    Ma, Mw, Sa, Sw = bits(a != 0), bits(w != 0), bits(a < 0), bits(w < 0)
    assert acc.item() == _popc(Ma & Mw) - 2 * _popc(Ma & Mw & (Sa ^ Sw))


@pytest.mark.parametrize("ba,bw", list(product([1, 2, 3], [1, 2, 3])))
@pytest.mark.parametrize("stride,pad,k", [(1, 1, 3), (2, 1, 3), (1, 0, 1), (2, 0, 1), (2, 3, 7)])
def test_conv_matches_torch_float64(ba, bw, stride, pad, k):
    """The oracle's direct convolution of dequantized levels equals
    torch.nn.functional.conv2d in float64 (zero padding), scaled to integer
    units 2^(f_a + f_w)."""
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(ba * 10 + bw + k)
    x = r.standard_normal((2, 33, 9, 8)).astype(np.float32)
    w = r.standard_normal((5, 33, k, k)).astype(np.float32) * 0.7
    al = O.quantize(x, ba, DEFAULT_THR[ba])
    wl = O.quantize(w, bw, DEFAULT_THR[bw])
    acc = O.conv2d_levels(al, wl, stride, pad, ba, bw)
    ref = torch.nn.functional.conv2d(torch.from_numpy(al), torch.from_numpy(wl),
                                     stride=stride, padding=pad).numpy()
    ref = ref * 2.0 ** (O.units_shift(ba) + O.units_shift(bw))
    assert np.array_equal(acc, ref.astype(np.int64))
    assert np.all(ref == np.round(ref))


def test_conv_brute_force_tiny():
    """Pure-Python loops on a tiny 3-bit x 3-bit case."""
    r = np.random.default_rng(4)
    lv = [0.0, 0.25, -0.25, 0.5, -0.5, 1.0, -1.0]
    a = r.choice(lv, (1, 3, 4, 5))
    w = r.choice(lv, (2, 3, 3, 3))
    acc = O.conv2d_levels(a, w, 1, 1, 3, 3)
    for o, y, x in product(range(2), range(4), range(5)):
        s = 0.0
        for c, ky, kx in product(range(3), range(3), range(3)):
            yi, xi = y - 1 + ky, x - 1 + kx
            if 0 <= yi < 4 and 0 <= xi < 5:
                s += a[0, c, yi, xi] * w[o, c, ky, kx]
        assert acc[0, o, y, x] == int(s * 16)


def test_zero_padding_of_binary_map():
    """Zero padding of a +-1 map contributes nothing: all +1 activations and
    weights give 4C at corners, 6C on edges and 9C inside (3x3, pad 1)."""
    C = 37
    a = np.ones((1, C, 5, 6))
    w = np.ones((1, C, 3, 3))
    acc = O.conv2d_levels(a, w, 1, 1, 1, 1)[0, 0]
    expect = np.full((5, 6), 9 * C)
    expect[0, :] = expect[-1, :] = 6 * C
    expect[:, 0] = expect[:, -1] = 6 * C
    expect[0, 0] = expect[0, -1] = expect[-1, 0] = expect[-1, -1] = 4 * C
    assert np.array_equal(acc, expect)


def test_non_integral_is_rejected():
    a = np.full((1, 1, 1, 1), 0.25)
    w = np.full((1, 1, 1, 1), 0.25)
    with pytest.raises(ArithmeticError):
        O.conv2d_levels(a, w, 1, 0, 1, 1)   # 1/16 claimed to be 1-bit units
