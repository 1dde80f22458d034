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


def _bf16_torch(x):
    """bf16 rounding by torch's conversion (independent of the oracle's)."""
    torch = pytest.importorskip("torch")
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16).float().numpy()


@pytest.mark.parametrize("last", [False, True])
def test_fc_train_step_wiring(last):
    """The composed step against properties it must have, at the paper's
    precision (fp32 operands): a_pre is the fp32 rounding of the exact
    (rational) product of the fp32 input and the fp32 weight AQE; g_in and the
    weight step are the gradients of sum(g~ * a~) with respect to the input
    and the weights (central differences in fp64), so a transposed or swapped
    operand fails; the last layer passes g through unmasked; a given a_pre
    replaces the forward product for every later stage."""
    r = np.random.default_rng(11)
    B, K, O_ = 3, 8, 4
    A = np.clip(r.standard_normal((B, K)), -1.5, 1.5).astype(np.float32)
    W = r.uniform(-1, 1, (O_, K)).astype(np.float32)
    G = (r.standard_normal((B, O_)) * 0.5).astype(np.float32)
    alpha, lr = 0.6, 0.125
    q_a = None if last else (2, DEFAULT_THR[2])
    a_out, g_in, W_new, a_pre = O.fc_train_step(A, W, G, alpha, lr, 1, DEFAULT_THR[1], q_a)
    Wh = O.aqe_forward_f32(W, alpha, 1, DEFAULT_THR[1])
    for i in range(B):
        for o in range(O_):
            exact = sum(Fraction(float(A[i, k])) * Fraction(float(Wh[o, k])) for k in range(K))
            assert a_pre[i, o] == np.float32(float(exact))
    if last:
        assert np.array_equal(a_out, a_pre)
        gt = G
    else:
        assert np.array_equal(a_out, O.aqe_forward_f32(a_pre, alpha, 2, DEFAULT_THR[2]))
        gt = O.aqe_backward_f32(a_pre, G, alpha)
    g64 = gt.astype(np.float64)
    L = lambda A_, W_: np.sum(g64 * (A_ @ W_.T))
    h = 1e-3
    A64, W64 = A.astype(np.float64), Wh.astype(np.float64)
    for i in range(B):
        for k in range(K):
            E = np.zeros_like(A64); E[i, k] = h
            d = (L(A64 + E, W64) - L(A64 - E, W64)) / (2 * h)
            assert abs(g_in[i, k] - d) <= 1e-6 * (1 + abs(d))
    for o in range(O_):
        for k in range(K):
            E = np.zeros_like(W64); E[o, k] = h
            d = (L(A64, W64 + E) - L(A64, W64 - E)) / (2 * h)
            want = np.clip(W[o, k] - lr * 2 * alpha * d, -1.0, 1.0)     # |W| <= 1: the mask passes
            assert abs(W_new[o, k] - want) <= 1e-6
    # a substituted forward product drives the later stages
    sub = (a_pre + np.float32(0.25)).astype(np.float32)
    a2, g2, W2, p2 = O.fc_train_step(A, W, G, alpha, lr, 1, DEFAULT_THR[1], q_a, a_pre=sub)
    assert np.array_equal(p2, sub)
    if not last:
        assert np.array_equal(a2, O.aqe_forward_f32(sub, alpha, 2, DEFAULT_THR[2]))
        g2t = O.aqe_backward_f32(sub, G, alpha).astype(np.float64)
        assert np.allclose(g2, g2t @ W64, rtol=2.0 ** -22, atol=1e-30)


def test_fc_train_step_full_precision():
    """The step keeps full precision: weights and inputs that bf16 cannot
    represent (1 + 2^-12, 1 + 2^-20) give the fp32 rounding of the exact
    product, not of a product of rounded operands."""
    A = np.full((1, 64), 1.0 + 2.0 ** -12, dtype=np.float32)
    W = np.full((2, 64), 0.5 + 2.0 ** -20, dtype=np.float32)
    G = np.ones((1, 2), dtype=np.float32)
    a_out, g_in, W_new, a_pre = O.fc_train_step(A, W, G, 0.0, 0.0, 1, DEFAULT_THR[1], None)
    exact = 64 * Fraction(float(A[0, 0])) * Fraction(float(W[0, 0]))
    assert a_pre[0, 0] == np.float32(float(exact)) and a_pre[0, 0] != np.float32(32.0)
    assert g_in[0, 0] == np.float32(float(2 * Fraction(float(W[0, 0]))))


def test_fc_train_step_alpha_zero():
    """alpha = 0: W^ = W, the masks' factor 2 alpha vanishes, so the weights
    stay as they are and (hidden layer) the input gradient is zero."""
    r = np.random.default_rng(12)
    A = r.standard_normal((4, 16)).astype(np.float32)
    W = r.uniform(-1, 1, (5, 16)).astype(np.float32)
    G = r.standard_normal((4, 5)).astype(np.float32)
    a_out, g_in, W_new, a_pre = O.fc_train_step(A, W, G, 0.0, 0.5, 2, DEFAULT_THR[2], (1, DEFAULT_THR[1]))
    assert np.array_equal(W_new, W)
    assert not g_in.any()
    assert np.array_equal(a_out, a_pre)


def test_bf16_round_array_matches_scalar():
    """The array form of the oracle's bf16 rounding equals its scalar form,
    ties and specials included."""
    x = np.concatenate([_x(seed=21), np.array([1.00390625, 1.01171875, -2.0 ** -130, 3.0e38, np.inf, -np.inf],
                                              dtype=np.float32)]).astype(np.float32)
    got = O.bf16_round(x)
    want = np.array([O.bf16_round_scalar(v) for v in x], dtype=np.float32)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("stride,pad,k", [(1, 1, 3), (2, 1, 3), (1, 0, 1), (2, 0, 2)])
def test_conv_backward_products_match_autograd(stride, pad, k):
    """The convolutional layer's input and weight gradients equal torch's
    autograd of conv2d in float64 (an independent implementation), strided
    and padded; a transposed or flipped kernel fails."""
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(100 + stride * 10 + pad + k)
    B, C, H, W, O_ = 2, 3, 7, 6, 4
    a = r.standard_normal((B, C, H, W))
    w = r.standard_normal((O_, C, k, k))
    at = torch.tensor(a, requires_grad=True)
    wt = torch.tensor(w, requires_grad=True)
    y = torch.nn.functional.conv2d(at, wt, stride=stride, padding=pad)
    g = r.standard_normal(tuple(y.shape))
    (y * torch.tensor(g)).sum().backward()
    assert np.allclose(O.conv2d_real(a, w, stride, pad), y.detach().numpy(), rtol=1e-12, atol=1e-12)
    assert np.allclose(O.conv2d_input_grad(g, w, stride, pad, H, W), at.grad.numpy(), rtol=1e-12, atol=1e-12)
    assert np.allclose(O.conv2d_weight_grad(g, a, k, k, stride, pad), wt.grad.numpy(), rtol=1e-12, atol=1e-12)


def test_conv_train_step_reduces_to_fc():
    """A 1 x 1 convolution over 1 x 1 images is a fully connected layer: the
    convolutional step equals fc_train_step bit for bit."""
    r = np.random.default_rng(13)
    B, K, O_ = 4, 16, 6
    A = np.clip(r.standard_normal((B, K)), -1.5, 1.5).astype(np.float32)
    W = r.uniform(-1, 1, (O_, K)).astype(np.float32)
    G = (r.standard_normal((B, O_)) * 0.5).astype(np.float32)
    for q_a in [None, (2, DEFAULT_THR[2])]:
        fc = O.fc_train_step(A, W, G, 0.7, 0.25, 3, DEFAULT_THR[3], q_a)
        cv = O.conv_train_step(A[:, :, None, None], W[:, :, None, None], G[:, :, None, None], 0.7, 0.25, 3,
                               DEFAULT_THR[3], 1, 0, q_a)
        for x, y in zip(fc, cv):
            assert np.array_equal(x, y.reshape(x.shape))


def test_conv_train_step_gradients():
    """The convolutional step's forward product, input gradient and weight
    step are those of the fp32 operands at full precision: torch autograd of
    conv2d in float64 (an independent implementation) on the fp32 input and
    weight AQE, with the mask of Eq. weight and the clip on the latent
    weights."""
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(14)
    A = np.clip(r.standard_normal((2, 4, 6, 6)), -1.5, 1.5).astype(np.float32)
    W = r.uniform(-1.2, 1.2, (3, 4, 3, 3)).astype(np.float32)       # some |w| > 1: masked
    G = (r.standard_normal((2, 3, 3, 3)) * 0.5).astype(np.float32)
    alpha, lr = 0.5, 0.125
    a_out, g_in, W_new, a_pre = O.conv_train_step(A, W, G, alpha, lr, 2, DEFAULT_THR[2], 2, 1, (1, DEFAULT_THR[1]))
    Wq = torch.tensor(O.aqe_forward_f32(W, alpha, 2, DEFAULT_THR[2]).astype(np.float64), requires_grad=True)
    Aq = torch.tensor(A.astype(np.float64), requires_grad=True)
    y = torch.nn.functional.conv2d(Aq, Wq, stride=2, padding=1)
    assert np.allclose(a_pre, y.detach().numpy(), rtol=2.0 ** -23, atol=1e-30)
    gt = O.aqe_backward_f32(a_pre, G, alpha).astype(np.float64)
    (y * torch.tensor(gt)).sum().backward()
    assert np.allclose(g_in, Aq.grad.numpy(), rtol=2.0 ** -23, atol=1e-30)
    gw = Wq.grad.numpy()
    want = np.clip(W - lr * np.where(np.abs(W) <= 1.0, 2 * alpha * gw, 0.0), -1.0, 1.0)
    assert np.allclose(W_new, want, rtol=0, atol=1e-6)
    assert np.array_equal(W_new[np.abs(W) > 1.0], np.clip(W[np.abs(W) > 1.0], -1, 1))
