"""GPU parity of the library's kernels against the CPU oracle, through the
C ABI: AQE forward/backward, quantize + pack, weight packing, the quantized
convolution (all nine bit-width pairs, ragged tiles), the fused block
epilogue and the fp32 first layer."""
from itertools import product

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, aqe_problem, conv_problem  # noqa: E402
from tests._gpu import case_seed, assert_close, dev_tensor, planes_view, words  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available(), "the GPU tests need a CUDA device"
    return torch.device("cuda:0")


@pytest.fixture(scope="module")
def M(dev):
    from paper_2003_04296_gb300 import minw
    return minw


# ------------------------------------------------------------------ AQE ----

@pytest.mark.parametrize("n", [0, 1, 7, 4096, 1000003])
@pytest.mark.parametrize("bits,alpha", [(1, 0.75), (2, 0.3), (3, 1.0), (1, 0.0)])
def test_aqe_forward(dev, M, n, bits, alpha):
    p = aqe_problem(100 + n, n)
    x = dev_tensor(p["x"], dev)
    y = torch.empty_like(x)
    M.aqe_forward(x, y, alpha, M.quant(bits, DEFAULT_THR[bits]))
    ref = O.aqe_forward(p["x"], alpha, bits, DEFAULT_THR[bits])
    assert_close(y.cpu().numpy(), ref)


@pytest.mark.parametrize("n", [0, 3, 4096, 1000003])
@pytest.mark.parametrize("alpha", [0.5, 0.75])
def test_aqe_backward(dev, M, n, alpha):
    p = aqe_problem(200 + n, n)
    x, g = dev_tensor(p["x"], dev), dev_tensor(p["g"], dev)
    gx = torch.empty_like(x)
    M.aqe_backward(x, g, gx, alpha)
    assert_close(gx.cpu().numpy(), O.aqe_backward(p["x"], p["g"], alpha))


PACK_SHAPES = [(2, 64, 8, 8), (3, 45, 5, 7), (2, 32, 4, 8), (1, 96, 14, 14), (1, 7, 1, 1)]


@pytest.mark.parametrize("shape", PACK_SHAPES)
@pytest.mark.parametrize("bits", [1, 2, 3])
def test_quantize_pack_fused(dev, M, shape, bits):
    B, C, H, W = shape
    x_np = (np.random.default_rng(B * C + H * W + bits).standard_normal(shape) * 1.2).astype(np.float32)
    x = dev_tensor(x_np, dev)
    planes = torch.full((M.packed_words(B, C, H, W, bits),), -1, dtype=torch.int32, device=dev)
    y = torch.empty_like(x)
    n = x.numel()
    mask = torch.full(((n + 31) // 32,), -1, dtype=torch.int32, device=dev)
    M.aqe_quantize_pack(x, M.quant(bits, DEFAULT_THR[bits]), planes, alpha=0.6, y=y, mask=mask)
    lv = O.quantize(x_np, bits, DEFAULT_THR[bits])
    assert np.array_equal(planes_view(planes, B, H, W, bits, C), O.pack(lv, bits))
    assert_close(y.cpu().numpy(), O.aqe_forward(x_np, 0.6, bits, DEFAULT_THR[bits]))
    bitsref = (np.abs(x_np.ravel()) <= 1.0).astype(np.uint64)
    got = words(mask)
    unpacked = (got[np.arange(n) // 32] >> (np.arange(n) % 32).astype(np.uint32)) & 1
    assert np.array_equal(unpacked.astype(np.uint64), bitsref)
    # masked backward consumes the packed mask
    g_np = np.random.default_rng(7).standard_normal(shape).astype(np.float32)
    gx = torch.empty_like(x)
    M.aqe_backward_masked(mask, dev_tensor(g_np, dev), gx, 0.6)
    assert_close(gx.cpu().numpy(), O.aqe_backward(x_np, g_np, 0.6))


def test_quantize_pack_scale(dev, M):
    x_np = np.random.default_rng(3).standard_normal((2, 64, 4, 4)).astype(np.float32)
    q = M.quant(3, DEFAULT_THR[3], scale=0.37)
    planes = torch.empty(M.packed_words(2, 64, 4, 4, 3), dtype=torch.int32, device=dev)
    M.aqe_quantize_pack(dev_tensor(x_np, dev), q, planes)
    lv = O.quantize(x_np, 3, DEFAULT_THR[3], np.full(2, 0.37, dtype=np.float32))
    assert np.array_equal(planes_view(planes, 2, 4, 4, 3, 64), O.pack(lv, 3))


@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("shape", [(70, 64, 3, 3), (10, 45, 1, 1), (5, 512, 4, 4)])
def test_pack_weights(dev, M, bits, shape):
    w_np = np.random.default_rng(sum(shape) + bits).normal(0, 0.05, shape).astype(np.float32)
    cs = (1.0 / np.abs(w_np.reshape(shape[0], -1)).max(1)).astype(np.float32)
    planes = torch.empty(M.packed_words(shape[0], shape[1], shape[2], shape[3], bits), dtype=torch.int32,
                         device=dev)
    M.minw_pack_weights(dev_tensor(w_np, dev), M.quant(bits, DEFAULT_THR[bits]), planes,
                        channel_scale=dev_tensor(cs, dev))
    lv = O.quantize(w_np, bits, DEFAULT_THR[bits], cs)
    assert np.array_equal(planes_view(planes, shape[0], shape[2], shape[3], bits, shape[1]), O.pack(lv, bits))


# ------------------------------------------------------------ convolution --

CONV_CASES = [
    # B, C, H, W, O, k, stride, pad
    (2, 64, 9, 7, 70, 3, 1, 1),      # ragged pixel tile, ragged channel tile
    (1, 128, 8, 8, 64, 3, 2, 1),     # stride 2
    (3, 32, 5, 5, 10, 1, 1, 0),      # 1x1, O < 32
    (2, 96, 6, 6, 33, 3, 1, 1),      # 3 words per pixel
    (4, 64, 4, 4, 20, 4, 1, 0),      # fully connected as a 4x4 convolution
    (2, 64, 1, 1, 130, 1, 1, 0),     # 1x1 spatial
]


def _conv_gpu(dev, M, p, variant, want_y=True):
    B, C, H, W, O_ = p["B"], p["C"], p["H"], p["W"], p["O"]
    ba, bw = p["bits_a"], p["bits_w"]
    act = torch.empty(M.packed_words(B, C, H, W, ba), dtype=torch.int32, device=dev)
    wgt = torch.empty(M.packed_words(O_, C, p["kh"], p["kw"], bw), dtype=torch.int32, device=dev)
    M.aqe_quantize_pack(dev_tensor(p["x"], dev), M.quant(ba, p["thr_a"]), act)
    M.minw_pack_weights(dev_tensor(p["w"], dev), M.quant(bw, p["thr_w"]), wgt,
                        channel_scale=dev_tensor(p["w_scale"], dev))
    Ho = (H + 2 * p["pad"] - p["kh"]) // p["stride"] + 1
    Wo = (W + 2 * p["pad"] - p["kw"]) // p["stride"] + 1
    acc = torch.full((B, O_, Ho, Wo), -7, dtype=torch.int32, device=dev)
    y = torch.empty((B, O_, Ho, Wo), dtype=torch.float32, device=dev) if want_y else None
    M.minw_conv2d(act, B, C, H, W, ba, wgt, O_, p["kh"], p["kw"], bw, p["stride"], p["pad"], acc_out=acc,
                  scale=dev_tensor(p["scale"], dev), shift=dev_tensor(p["shift"], dev), y_out=y,
                  variant=variant)
    return act, wgt, acc, y


def _conv_ref(p):
    al = O.quantize(p["x"], p["bits_a"], p["thr_a"])
    wl = O.quantize(p["w"], p["bits_w"], p["thr_w"], p["w_scale"])
    return O.conv2d_levels(al, wl, p["stride"], p["pad"], p["bits_a"], p["bits_w"])


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("ba,bw", list(product([1, 2, 3], [1, 2, 3])))
def test_conv2d_popc(dev, M, case, ba, bw):
    B, C, H, W, O_, k, s, pad = case
    p = conv_problem(case_seed(case, ba, bw), B, C, H, W, O_, k, k, s, pad, ba, bw, w_sigma=0.5)
    _, _, acc, y = _conv_gpu(dev, M, p, M.VARIANT_POPC)
    ref = _conv_ref(p)
    assert np.array_equal(acc.cpu().numpy(), ref)
    assert np.array_equal(y.cpu().numpy(), O.affine(ref, p["scale"], p["shift"]))


@pytest.mark.parametrize("ba,bw", [(1, 1), (2, 2), (3, 3), (2, 1)])
def test_conv_block_pool_quantize(dev, M, ba, bw):
    B, C, H, W, O_ = 2, 64, 16, 16, 96
    p = conv_problem(31 + ba * 3 + bw, B, C, H, W, O_, 3, 3, 1, 1, ba, bw, w_sigma=0.5)
    act = torch.empty(M.packed_words(B, C, H, W, ba), dtype=torch.int32, device=dev)
    wgt = torch.empty(M.packed_words(O_, C, 3, 3, bw), dtype=torch.int32, device=dev)
    M.aqe_quantize_pack(dev_tensor(p["x"], dev), M.quant(ba, p["thr_a"]), act)
    M.minw_pack_weights(dev_tensor(p["w"], dev), M.quant(bw, p["thr_w"]), wgt,
                        channel_scale=dev_tensor(p["w_scale"], dev))
    bo = ba
    planes = torch.full((M.packed_words(B, O_, 8, 8, bo),), -1, dtype=torch.int32, device=dev)
    y = torch.empty((B, O_, 8, 8), dtype=torch.float32, device=dev)
    M.minw_conv_block(act, B, C, H, W, ba, wgt, O_, 3, 3, bw, 1, 1, 1, dev_tensor(p["scale"], dev),
                      dev_tensor(p["shift"], dev), q_out=M.quant(bo, DEFAULT_THR[bo]), planes_out=planes,
                      y_out=y, variant=M.VARIANT_POPC)
    acc = O.maxpool_i32(_conv_ref(p), 2, 2)
    yr = O.hardtanh(O.affine(acc, p["scale"], p["shift"]))
    assert np.array_equal(y.cpu().numpy(), yr)
    lv = O.quantize(yr, bo, DEFAULT_THR[bo])
    assert np.array_equal(planes_view(planes, B, 8, 8, bo, O_), O.pack(lv, bo))


@pytest.mark.parametrize("bits_w,bits_out", [(1, 1), (2, 2), (3, 3)])
def test_conv_first(dev, M, bits_w, bits_out):
    B, C, H, W, O_ = 3, 3, 11, 9, 40
    r = np.random.default_rng(bits_w)
    x = r.uniform(-1, 1, (B, C, H, W)).astype(np.float32)
    w = r.normal(0, 0.05, (O_, C, 3, 3)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32)
    scale = (r.normal(1, 0.1, O_) / np.sqrt(27.0)).astype(np.float32)
    shift = r.normal(0, 0.1, O_).astype(np.float32)
    planes = torch.empty(M.packed_words(B, O_, H, W, bits_out), dtype=torch.int32, device=dev)
    y = torch.empty((B, O_, H, W), dtype=torch.float32, device=dev)
    M.minw_conv_first(dev_tensor(x, dev), dev_tensor(w, dev), 1, 1, dev_tensor(scale, dev),
                      dev_tensor(shift, dev), q_w=M.quant(bits_w, DEFAULT_THR[bits_w]),
                      channel_scale=dev_tensor(cs, dev), q_out=M.quant(bits_out, DEFAULT_THR[bits_out]),
                      planes_out=planes, y_out=y)
    wl = O.quantize(w, bits_w, DEFAULT_THR[bits_w], cs).astype(np.float32)
    yr = O.hardtanh(O.affine(O.conv2d_f32_seq(x, wl, 1, 1), scale, shift))
    assert np.array_equal(y.cpu().numpy(), yr)
    lv = O.quantize(yr, bits_out, DEFAULT_THR[bits_out])
    assert np.array_equal(planes_view(planes, B, H, W, bits_out, O_), O.pack(lv, bits_out))


@pytest.mark.parametrize("quant_w", [True, False])
def test_conv_first_strided_stem(dev, M, quant_w):
    """A 7x7 / stride 2 / pad 3 first layer (ResNet stem shape) on a ragged
    23x23 image, with quantized or fp32 weights."""
    B, C, H, W, O_, k = 2, 3, 23, 23, 64, 7
    r = np.random.default_rng(17)
    x = r.standard_normal((B, C, H, W)).astype(np.float32)
    w = r.normal(0, 0.05, (O_, C, k, k)).astype(np.float32)
    scale = (r.normal(1, 0.1, O_) / np.sqrt(147.0)).astype(np.float32)
    shift = r.normal(0, 0.1, O_).astype(np.float32)
    if quant_w:
        cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32)
        wl = O.quantize(w, 3, DEFAULT_THR[3], cs).astype(np.float32)
        kw_ = dict(q_w=M.quant(3, DEFAULT_THR[3]), channel_scale=dev_tensor(cs, dev))
    else:
        wl = w
        kw_ = {}
    Ho = (H + 6 - k) // 2 + 1
    planes = torch.empty(M.packed_words(B, O_, Ho, Ho, 2), dtype=torch.int32, device=dev)
    y = torch.empty((B, O_, Ho, Ho), dtype=torch.float32, device=dev)
    M.minw_conv_first(dev_tensor(x, dev), dev_tensor(w, dev), 2, 3, dev_tensor(scale, dev), dev_tensor(shift, dev),
                      q_out=M.quant(2, DEFAULT_THR[2]), planes_out=planes, y_out=y, **kw_)
    yr = O.hardtanh(O.affine(O.conv2d_f32_seq(x, wl, 2, 3), scale, shift))
    assert np.array_equal(y.cpu().numpy(), yr)
    lv = O.quantize(yr, 2, DEFAULT_THR[2])
    assert np.array_equal(planes_view(planes, B, Ho, Ho, 2, O_), O.pack(lv, 2))


def test_conv2d_adversarial_magnitudes(dev, M):
    """Largest accumulators of the bench shapes: every 3-bit level at +-1 on a
    512-channel 3x3 kernel (|acc| = 16 * 4608) next to small products."""
    B, C, H, W, O_ = 2, 512, 6, 6, 64
    x = np.ones((B, C, H, W), dtype=np.float32)
    x[:, :, ::2, :] = -1.0
    x[1, :256] = 0.2                          # 1/4 levels (1 unit) after a large pair
    w = np.ones((O_, C, 3, 3), dtype=np.float32)
    w[::2] = -1.0
    w[:, ::7] *= 0.45                          # 1/2 levels
    p = dict(x=x, w=w, w_scale=np.ones(O_, np.float32), thr_a=DEFAULT_THR[3], thr_w=DEFAULT_THR[3],
             scale=np.ones(O_, np.float32), shift=np.zeros(O_, np.float32), B=B, C=C, H=H, W=W, O=O_,
             kh=3, kw=3, stride=1, pad=1, bits_a=3, bits_w=3)
    for variant in (M.VARIANT_POPC,):
        _, _, acc, _ = _conv_gpu(dev, M, p, variant)
        assert np.array_equal(acc.cpu().numpy(), _conv_ref(p))
