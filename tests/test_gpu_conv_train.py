"""GPU parity of Algorithm 1's training step on a convolutional layer
(minw_conv_train_step), through the C ABI, against the oracle's step at the
paper's precision (oracle.conv_train_step: fp32 operands, fp64 sums).

The GPU forms its three products -- the forward convolution, the input
gradient (the transposed convolution) and the weight gradient (the
correlation over the batch and the image) -- from bf16 roundings of the fp32
operands with fp32 accumulation, so each product P * Q with K terms per
output differs from the exact one by at most

    (2^-7 + 2^-16 + K 2^-23 (1 + 2^-8)^2) (|P| * |Q|) + 2^-24 |P * Q|

(two operand roundings of relative size 2^-8, the fp32 accumulation in any
order, split slices included, and the oracle's own rounding to fp32), where
|P| * |Q| is the same product of the absolute values.  The stages after the
forward product are compared with the oracle fed the GPU's forward product
(its a_pre argument): a_out bit for bit, g_in within the bound, the updated
weights within lr 2 alpha times the weight gradient's bound plus one fp32
ulp.  Shapes cover strides 1 and 2, a stride that leaves input rows unread,
output channels that are not a multiple of 64, 1 x 1 kernels, and a weight
gradient long enough to be split along the pixels."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR  # noqa: E402
from tests._gpu import dev_tensor  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()
    return torch.device("cuda:0")


@pytest.fixture(scope="module")
def M(dev):
    from paper_2003_04296_gb300 import minw
    return minw


def _problem(seed, B, C, H, W, O_, k, stride, pad):
    r = np.random.default_rng(seed)
    Ho, Wo = (H + 2 * pad - k) // stride + 1, (W + 2 * pad - k) // stride + 1
    A = np.clip(r.standard_normal((B, C, H, W)), -1.5, 1.5).astype(np.float32)
    Wt = r.uniform(-1, 1, (O_, C, k, k)).astype(np.float32)
    G = (r.standard_normal((B, O_, Ho, Wo)) * 0.1).astype(np.float32)
    return A, Wt, G


def _coef(K):
    return 2.0 ** -7 + 2.0 ** -16 + K * 2.0 ** -23 * (1 + 2.0 ** -8) ** 2


def _within(got, ref, bound, what):
    err = np.abs(got.astype(np.float64) - ref.astype(np.float64))
    assert (err <= bound).all(), f"{what}: worst err/bound {np.max(err / bound)}"


CASES = [
    # B, C, H, W, O, k, stride, pad, alpha, bits_w, bits_a
    (8, 64, 8, 8, 64, 3, 1, 1, 0.75, 1, 1),
    (4, 128, 16, 16, 96, 3, 2, 1, 0.5, 2, 2),      # stride 2, O % 64 != 0
    (4, 64, 10, 10, 40, 3, 2, 0, 0.3, 3, 1),       # stride 2 leaves the last input row and column unread
    (16, 64, 4, 4, 128, 1, 1, 0, 0.6, 1, 2),       # 1 x 1 kernel
    (16, 128, 16, 16, 128, 3, 1, 1, 0.75, 1, 1),   # 4096 pixels: the weight gradient splits along them
]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("last", [False, True])
def test_conv_train_step(dev, M, case, last):
    B, C, H, W, O_, k, stride, pad, alpha, bw, ba = case
    lr = 0.05
    A, Wl, G = _problem(11 + B + C + O_ + k + stride, B, C, H, W, O_, k, stride, pad)
    Ho, Wo = G.shape[2], G.shape[3]
    qw, qa = M.quant(bw, DEFAULT_THR[bw]), (None if last else M.quant(ba, DEFAULT_THR[ba]))
    q_a = None if last else (ba, DEFAULT_THR[ba])
    At, Gt = dev_tensor(A, dev), dev_tensor(G, dev)
    ws = torch.empty(M.minw_conv_train_workspace_bytes(B, C, H, W, O_, k, k, stride, pad), dtype=torch.uint8,
                     device=dev)
    outs = []
    for _ in range(2):
        W1 = dev_tensor(Wl, dev)
        a1 = torch.empty((B, O_, Ho, Wo), device=dev)
        g1 = torch.empty((B, C, H, W), device=dev)
        pre = torch.empty((B, O_, Ho, Wo), device=dev)
        M.minw_conv_train_step(At, W1, Gt, stride, pad, alpha, lr, qw, qa, a1, g1, ws, a_pre=pre)
        torch.cuda.synchronize()
        outs.append((W1.cpu().numpy(), a1.cpu().numpy(), g1.cpu().numpy(), pre.cpu().numpy()))
    assert M.minw_get_last_device_error() == M.MINW_OK
    W1, a1, g1, pre = outs[0]
    for x, y in zip(outs[0], outs[1][:3]):
        assert np.array_equal(x, y)          # fixed summation order: the same bits on every call
    at = a1 if last else pre
    what = O.aqe_forward_f32(Wl, alpha, bw, DEFAULT_THR[bw])
    # the forward product against the paper-precision oracle's
    ref = O.conv_train_step(A, Wl, G, alpha, lr, bw, DEFAULT_THR[bw], stride, pad, q_a)
    a64 = np.abs(A).astype(np.float64)
    w64 = np.abs(what).astype(np.float64)
    mag_f = O.conv2d_real(a64, w64, stride, pad)
    _within(at, ref[3], _coef(C * k * k) * mag_f + 2.0 ** -24 * np.abs(ref[3]) + 1e-30, "a~")
    # the later stages with the GPU's a~ substituted
    a_ref, gin_ref, W_ref, _ = O.conv_train_step(A, Wl, G, alpha, lr, bw, DEFAULT_THR[bw], stride, pad, q_a,
                                                 a_pre=at)
    if not last:
        assert np.array_equal(a1, a_ref)
    gat = G if last else O.aqe_backward_f32(at, G, alpha)
    g64 = np.abs(gat).astype(np.float64)
    Op = (O_ + 63) // 64 * 64
    mag_in = O.conv2d_input_grad(g64, w64, stride, pad, H, W)
    _within(g1, gin_ref, _coef(Op * k * k) * mag_in + 2.0 ** -24 * np.abs(gin_ref) + 1e-30, "g_in")
    mag_w = O.conv2d_weight_grad(g64, a64, k, k, stride, pad)
    gw_ref = O.conv2d_weight_grad(gat.astype(np.float64), A.astype(np.float64), k, k, stride, pad)
    gbound = _coef(B * Ho * Wo) * mag_w + 2.0 ** -24 * np.abs(gw_ref)
    _within(W1, W_ref, lr * 2 * alpha * (gbound + 2.0 ** -24 * np.abs(gw_ref)) + 2.0 ** -23, "W")
    assert np.abs(W1).max() <= 1.0


def test_conv_train_step_alpha_zero(dev, M):
    """alpha = 0 (the start of the schedule, no quantization): the step
    leaves W unchanged (the mask of Eq. weight carries the factor 2 alpha),
    the input gradient is zero (so is g~), and a_out equals a~ (Eq. activation
    at alpha = 0 is the identity)."""
    B, C, H, W, O_, k = 8, 64, 8, 8, 64, 3
    A, Wl, G = _problem(5, B, C, H, W, O_, k, 1, 1)
    ws = torch.empty(M.minw_conv_train_workspace_bytes(B, C, H, W, O_, k, k, 1, 1), dtype=torch.uint8, device=dev)
    W1 = dev_tensor(Wl, dev)
    a1, g1, pre = (torch.empty((B, O_, H, W), device=dev), torch.empty((B, C, H, W), device=dev),
                   torch.empty((B, O_, H, W), device=dev))
    M.minw_conv_train_step(dev_tensor(A, dev), W1, dev_tensor(G, dev), 1, 1, 0.0, 0.1, M.quant(1), M.quant(1), a1,
                           g1, ws, a_pre=pre)
    torch.cuda.synchronize()
    assert np.array_equal(W1.cpu().numpy(), Wl)
    assert not g1.cpu().numpy().any()
    assert np.array_equal(a1.cpu().numpy(), pre.cpu().numpy())


def test_conv_train_step_errors(dev, M):
    A = torch.zeros((2, 32, 8, 8), device=dev)
    W = torch.zeros((64, 32, 3, 3), device=dev)
    G = torch.zeros((2, 64, 8, 8), device=dev)
    ws = torch.empty(1 << 20, dtype=torch.uint8, device=dev)
    out = torch.empty((2, 64, 8, 8), device=dev)
    with pytest.raises(M.MinwError):          # C % 64 != 0
        M.minw_conv_train_step(A, W, G, 1, 1, 0.5, 0.1, M.quant(1), None, out, None, ws)
    A = torch.zeros((1, 64, 4, 4), device=dev)
    W = torch.zeros((64, 64, 3, 3), device=dev)
    G = torch.zeros((1, 64, 4, 4), device=dev)
    out = torch.empty((1, 64, 4, 4), device=dev)
    with pytest.raises(M.MinwError):          # B Ho Wo = 16 is not a multiple of 64
        M.minw_conv_train_step(A, W, G, 1, 1, 0.5, 0.1, M.quant(1), None, out, None, ws)
    assert M.minw_conv_train_workspace_bytes(1, 64, 4, 4, 64, 3, 3, 3, 1) == 0     # stride 3
