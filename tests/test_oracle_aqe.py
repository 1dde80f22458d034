"""Pins of the oracle's AQE forward/backward (Eq. ours, Eq. activation,
Eq. weight) against the limits, theorems and derivatives the paper states."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2003_04296_gb300.inputs import DEFAULT_THR


def _x(n=5001, seed=0):
    r = np.random.default_rng(seed)
    return np.concatenate([r.standard_normal(n) * 1.5, [0.0, 1.0, -1.0, 0.5, -0.75]]).astype(np.float32)


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_alpha_limits(bits):
    """Eq. ours: alpha = 1 gives the quantized neuron h(a), alpha = 0 the identity."""
    x = _x()
    thr = DEFAULT_THR[bits]
    assert np.array_equal(O.aqe_forward(x, 1.0, bits, thr), O.quantize(x[None], bits, thr)[0])
    assert np.array_equal(O.aqe_forward(x, 0.0, bits, thr), x.astype(np.float64))


@pytest.mark.parametrize("alpha", [0.1, 0.5, 0.9])
def test_distance_to_h_shrinks_by_one_minus_alpha(alpha):
    """|h^ - h| = (1 - alpha) |a - h| (Eq. ours), so h^ -> h as alpha -> 1."""
    x = _x()
    hq = O.quantize(x[None], 3, DEFAULT_THR[3])[0]
    y = O.aqe_forward(x, alpha, 3, DEFAULT_THR[3])
    np.testing.assert_allclose(np.abs(y - hq), (1 - alpha) * np.abs(x - hq), rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("alpha", [0.05, 0.3, 0.5, 0.8])
def test_theorem3_geometric_series(alpha):
    """Theorem 3: iterating a(n+1) = h^(a(n)) gives
    a(n+1) = (1 - alpha)^n a(1) + h (1 - (1 - alpha)^n) and tends to h = sign(a(1))."""
    a1 = np.array([0.3, -0.7, 2.5, -1.9, 0.01], dtype=np.float32)
    a = a1.astype(np.float64)
    hs = np.where(a1 > 0, 1.0, -1.0)
    for n in range(1, 40):
        a = O.aqe_forward(a.astype(np.float32), alpha, 1)
        closed = (1 - alpha) ** n * a1 + hs * (1 - (1 - alpha) ** n)
        # the oracle takes fp32 inputs: one fp32 rounding per step
        np.testing.assert_allclose(a, closed, rtol=0, atol=1e-6 * n)
    if alpha >= 0.3:
        np.testing.assert_allclose(a, hs, atol=1e-5)


def test_stochastic_expectation_is_hardtanh():
    """Eq. our with z ~ U[-1, 1]: E_z[sign(a - z)] = max(-1, min(1, a)), the
    HardTanh of Sec. III-E; Monte Carlo within 5 sigma."""
    r = np.random.default_rng(11)
    n = 200000
    for a in [-1.7, -0.6, -0.1, 0.0, 0.25, 0.9, 1.3]:
        z = r.uniform(-1.0, 1.0, n)
        est = np.mean(np.where(a - z > 0, 1.0, -1.0))
        exact = O.hardtanh(np.array([a], dtype=np.float32))[0]
        sig = np.sqrt(max(1 - exact ** 2, 1e-12) / n)
        assert abs(est - exact) <= 5 * sig + 1e-12


@pytest.mark.parametrize("alpha", [0.25, 0.5, 0.75, 1.0])
def test_backward_matches_central_difference(alpha):
    """Eq. activation backward 2 alpha g 1[|a| <= 1] is the derivative of
    2 alpha g HardTanh(a) (Theorem 1, Eq. ste2; HardTanh is the function whose
    slope is 1[|a| <= 1], Sec. III-E).  Central differences of the oracle's own
    HardTanh, step 1e-4, away from the kinks at +-1."""
    r = np.random.default_rng(5)
    x = (r.standard_normal(4000) * 1.5).astype(np.float32)
    g = r.standard_normal(4000).astype(np.float32)
    h = 1e-4
    keep = np.abs(np.abs(x.astype(np.float64)) - 1.0) > 4 * h
    x, g = x[keep], g[keep]
    xd = x.astype(np.float64)

    def F(v):  # 2 alpha * HardTanh, with HardTanh evaluated in fp64 from its definition
        return 2 * alpha * np.maximum(-1.0, np.minimum(1.0, v))

    fd = (F(xd + h) - F(xd - h)) / (2 * h)
    gx = O.aqe_backward(x, g, alpha)
    ref = g.astype(np.float64) * fd
    np.testing.assert_allclose(gx, ref, rtol=1e-4, atol=1e-12)


def test_backward_mask_is_closed_interval():
    """Eq. activation uses 1[|a| <= 1]: a = +-1 still passes the gradient."""
    x = np.array([1.0, -1.0, np.nextafter(np.float32(1), np.float32(2)), -1.0000001], dtype=np.float32)
    g = np.ones(4, dtype=np.float32)
    assert list(O.aqe_backward(x, g, 0.5)) == [1.0, 1.0, 0.0, 0.0]


def test_half_alpha_is_ste():
    """Theorem 1: at alpha = 1/2 the AQE backward is the STE of Eq. ste,
    g 1[|a| <= 1]."""
    r = np.random.default_rng(9)
    x = (r.standard_normal(10000) * 1.2).astype(np.float32)
    g = r.standard_normal(10000).astype(np.float32)
    ste = np.where(np.abs(x) <= 1.0, g, 0.0).astype(np.float64)
    assert np.array_equal(O.aqe_backward(x, g, 0.5), ste)


def test_weight_form_is_same_rule():
    """Eq. weight applies the same forward and backward to latent weights."""
    w = np.random.default_rng(2).normal(0, 0.6, 3000).astype(np.float32)
    g = np.ones_like(w)
    gx = O.aqe_backward(w, g, 0.75)
    assert np.array_equal(gx, np.where(np.abs(w) <= 1, 1.5, 0.0))


# ---------------------------------------------------------------------------
# Stochastic AQE (Eq. our) with the counter-based generator
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("key,counter", [
    ((0x0123456789ABCDEF, 0xFEDCBA9876543210), (1, 0, 0, 0)),
    ((0, 0), (7, 0, 0, 0)),
    ((2**64 - 1, 2**64 - 1), (3, 2**64 - 1, 5, 2**63)),
    ((12345, 0), (0, 1, 0, 0)),            # numpy's carry from counter word 0 into word 1
])
def test_philox_matches_numpy(key, counter):
    """The oracle's Philox4x64-10 block equals numpy's Philox bit generator
    (same published algorithm; numpy advances its 256-bit counter by one
    before each block, so counter c comes from a generator started at c - 1)."""
    c = [int(v) for v in counter]
    prev = list(c)
    for w in range(4):                     # c - 1 with borrow across the four words
        if prev[w] > 0:
            prev[w] -= 1
            break
        prev[w] = 2**64 - 1
    bg = np.random.Philox(key=np.array(key, dtype=np.uint64), counter=np.array(prev, dtype=np.uint64))
    want = bg.random_raw(4)
    got = O.philox4x64_10(np.array(c, dtype=np.uint64), np.array(key, dtype=np.uint64))
    assert np.array_equal(got, want)


def test_noise_grid_and_uniformity():
    """z lies on the 2^-23 grid of [-1, 1) and is uniform: mean, variance and
    a 64-bin chi-square over 2^20 draws within their 5-sigma bounds."""
    n = 1 << 20
    _, z = O.aqe_forward_stochastic(np.zeros(n, dtype=np.float32), 0.5, seed=7, offset=0)
    z = z.astype(np.float64)
    assert z.min() >= -1.0 and z.max() < 1.0
    k = (z + 1.0) * 2.0 ** 23
    assert np.array_equal(k, np.rint(k))
    assert abs(z.mean()) < 5 * np.sqrt(1 / 3 / n)
    assert abs(z.var() - 1 / 3) < 5 * np.sqrt(4 / 45 / n)
    counts = np.histogram(z, bins=64, range=(-1.0, 1.0))[0]
    exp = n / 64
    chi2 = np.sum((counts - exp) ** 2 / exp)
    assert chi2 < 63 + 5 * np.sqrt(2 * 63)


@pytest.mark.parametrize("alpha", [0.25, 0.75])
def test_stochastic_theorem1_expectation(alpha):
    """Theorem 1's premise on the oracle's own draws: (h^ - (1 - alpha) a) / alpha
    = sign(a - z) averages to max(-1, min(1, a)) (Monte Carlo within 5 sigma),
    and each draw is exactly +-1 around the identity term."""
    m = 1 << 16
    for j, a in enumerate([-1.4, -0.5, 0.0, 0.3, 0.95, 2.0]):
        x = np.full(m, a, dtype=np.float32)
        y, z = O.aqe_forward_stochastic(x, alpha, seed=100 + j, offset=3)
        s = (y - (1.0 - alpha) * np.float64(np.float32(a))) / alpha
        np.testing.assert_allclose(np.abs(s), 1.0, rtol=0, atol=1e-9)
        assert np.array_equal(s > 0, x.astype(np.float64) > z)
        exact = float(np.clip(np.float32(a), -1.0, 1.0))
        sig = np.sqrt(max(1 - exact ** 2, 1e-12) / m)
        assert abs(s.mean() - exact) <= 5 * sig + 2.0 ** -22


def test_stochastic_limits_and_counter_layout():
    """alpha = 1 gives sign(a - z) in {-1, 1}, alpha = 0 the identity; element
    i at offset o draws the same noise as element i - 8k at offset o + k, and
    another seed draws other noise."""
    x = np.random.default_rng(3).standard_normal(1000).astype(np.float32)
    y1, z1 = O.aqe_forward_stochastic(x, 1.0, seed=9, offset=5)
    assert np.array_equal(np.abs(y1), np.ones_like(y1))
    y0, _ = O.aqe_forward_stochastic(x, 0.0, seed=9, offset=5)
    assert np.array_equal(y0, x.astype(np.float64))
    _, z2 = O.aqe_forward_stochastic(x[:1000 - 24], 1.0, seed=9, offset=5 + 3)
    assert np.array_equal(z2, z1[24:])
    _, z3 = O.aqe_forward_stochastic(x, 1.0, seed=10, offset=5)
    assert np.mean(z3 == z1) < 0.01


def test_stochastic_noise_words_follow_r18():
    """The noise of elements 8 c .. 8 c + 7 at offset o is the Philox4x64-10
    block at counter (o + c, 0, 0, 0), key (seed, 0) (the block pinned to
    numpy's generator above), split into its eight 32-bit words low half
    first, each mapped to (u >> 8) 2^-23 - 1: a swapped half, word or
    counter shows here though the noise statistics would not change."""
    seed, offset = 0x9E3779B97F4A7C15, 11
    _, z = O.aqe_forward_stochastic(np.zeros(24, dtype=np.float32), 0.5, seed=seed, offset=offset)
    for c in range(3):
        blk = O.philox4x64_10(np.array([offset + c, 0, 0, 0], dtype=np.uint64), np.array([seed, 0], dtype=np.uint64))
        words = []
        for w in blk:
            words += [int(w) & 0xFFFFFFFF, int(w) >> 32]
        want = np.array([(u >> 8) * 2.0 ** -23 - 1.0 for u in words], dtype=np.float32)
        assert np.array_equal(z[8 * c:8 * c + 8], want)
