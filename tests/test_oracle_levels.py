"""Pins of the oracle's quantizer h (Eq. sign, Eq. tnn, Eq. qnn; level sets of
Sec. IV-A) against hand-worked values and properties the paper fixes."""
import os

import numpy as np
import pytest

from oracle import oracle as O
from paper_2003_04296_gb300.inputs import DEFAULT_THR

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "levels.txt")

LEVEL_SETS = {1: {-1.0, 1.0}, 2: {-1.0, 0.0, 1.0},
              3: {0.0, 0.25, -0.25, 0.5, -0.5, 1.0, -1.0}}


def _golden_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            b, x, e = line.split()
            rows.append((int(b), float(x), float(e)))
    return rows


@pytest.mark.parametrize("bits,x,expected", _golden_rows())
def test_golden_levels(bits, x, expected):
    assert O.h(x, bits, DEFAULT_THR[bits]) == expected


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_level_set_membership_and_monotone(bits):
    x = np.sort(np.random.default_rng(1).standard_normal(20000).astype(np.float32) * 1.5)
    lv = O.quantize(x[None], bits, DEFAULT_THR[bits])[0]
    assert set(np.unique(lv)).issubset(LEVEL_SETS[bits])
    assert np.all(np.diff(lv) >= 0)                     # h is non-decreasing
    # every level of the set is reached on a wide input
    assert set(np.unique(lv)) == LEVEL_SETS[bits]


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_idempotent(bits):
    levels = np.array(sorted(LEVEL_SETS[bits]), dtype=np.float32)
    again = O.quantize(levels[None], bits, DEFAULT_THR[bits])[0]
    assert np.array_equal(again, levels.astype(np.float64))


@pytest.mark.parametrize("bits", [2, 3])
def test_threshold_neighbours(bits):
    """Just above each threshold the magnitude steps up; at it, it does not."""
    thr = [t for t in DEFAULT_THR[bits] if t > 0]
    for t in thr:
        t32 = np.float32(t)
        up = np.nextafter(t32, np.float32(np.inf))
        for s in (1.0, -1.0):
            lo = abs(O.h(s * t32, bits, DEFAULT_THR[bits]))
            hi = abs(O.h(s * up, bits, DEFAULT_THR[bits]))
            assert hi > lo


def test_qnn_reduces_to_tnn_and_sign():
    """Eq. qnn with n = 2 (q = 1 threshold) is Eq. tnn; with n = 1 (q = 0) it is Eq. sign."""
    xs = np.concatenate([np.linspace(-2, 2, 4001), [0.0, -0.0, 0.5, -0.5]])
    for x in xs:
        assert O.qnn(x, 2, [0.5]) == O.h(np.float32(x), 2, (0.5,))
        assert O.qnn(x, 1, []) == (1.0 if x > 0 else -1.0)


@pytest.mark.parametrize("n", [2, 3, 4])
def test_qnn_level_count(n):
    """An n-bit QNN has q = 2^(n-1)-1 magnitudes 2^-p (p = 0..q-1) plus zero,
    i.e. 2^n - 1 distinct levels."""
    q = 2 ** (n - 1) - 1
    mags = [2.0 ** -p for p in range(q)]
    # thresholds at midpoints between consecutive magnitudes (and half the smallest)
    thr = [(mags[i] + mags[i + 1]) / 2 for i in range(q - 1)] + [mags[-1] / 2]
    xs = np.linspace(-1.5, 1.5, 30001)
    vals = {O.qnn(x, n, thr) for x in xs}
    assert len(vals) == 2 ** n - 1
    assert vals == {0.0} | {s * m for m in mags for s in (1, -1)}


def test_scale_is_one_fp32_multiply():
    rng = np.random.default_rng(7)
    x = rng.standard_normal(2000).astype(np.float32)
    s = np.float32(3.3)
    for v in x[:200]:
        assert O.h(v, 3, DEFAULT_THR[3], s) == O.h(np.float32(v * s), 3, DEFAULT_THR[3], 1.0)


def test_per_channel_scale_quantize():
    w = np.random.default_rng(3).normal(0, 0.05, (4, 2, 3, 3)).astype(np.float32)
    s = (1.0 / np.abs(w.reshape(4, -1)).max(1)).astype(np.float32)
    lv = O.quantize(w, 3, DEFAULT_THR[3], s)
    # the largest-magnitude weight of every channel maps to +-1
    for o in range(4):
        i = np.argmax(np.abs(w[o]))
        assert abs(lv[o].ravel()[i]) == 1.0
