"""Pins of the oracle's weight-only pieces (full-precision activations times
1-3-bit weights, the XNOR / SHIFT ADDER layers of Sec. IV): the bf16 rounding
against torch's conversion, the fp64 real-valued convolution against
torch.nn.functional.conv2d in float64, and its agreement with the integer
convolution of levels."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2003_04296_gb300.inputs import DEFAULT_THR

torch = pytest.importorskip("torch")


def test_bf16_round_matches_torch():
    r = np.random.default_rng(0)
    x = np.concatenate([r.standard_normal(4000) * 10.0 ** r.integers(-6, 6, 4000),
                        [0.0, -0.0, 1.0, 1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -(1 + 2.0 ** -8), 3.0e38, -1.0e-40,
                         np.inf, -np.inf]]).astype(np.float32)
    got = O.bf16_round(x)
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("case", [(2, 5, 7, 6, 4, 3, 1, 1), (1, 3, 9, 9, 2, 3, 2, 1), (2, 4, 5, 5, 3, 1, 1, 0),
                                  (1, 2, 6, 8, 3, 3, 2, 0)])
def test_conv2d_real_matches_torch(case):
    B, C, H, W, O_, k, s, pad = case
    r = np.random.default_rng(sum(case))
    a = r.standard_normal((B, C, H, W))
    w = r.standard_normal((O_, C, k, k))
    got = O.conv2d_real(a, w, s, pad)
    want = torch.nn.functional.conv2d(torch.from_numpy(a), torch.from_numpy(w), stride=s, padding=pad).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_conv2d_real_on_levels_is_the_integer_product(bits):
    r = np.random.default_rng(bits)
    x = r.standard_normal((2, 32, 5, 6)).astype(np.float32)
    w = r.standard_normal((8, 32, 3, 3)).astype(np.float32)
    al = O.quantize(x, bits, DEFAULT_THR[bits])
    wl = O.quantize(w, bits, DEFAULT_THR[bits])
    acc = O.conv2d_levels(al, wl, 1, 1, bits, bits)
    sh = O.units_shift(bits) * 2
    assert np.array_equal(O.conv2d_real(al, wl, 1, 1) * 2.0 ** sh, acc.astype(np.float64))
