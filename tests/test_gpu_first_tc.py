"""GPU parity of the tensor-core first layer (fp16 split operands, an error
bound per output and the exact fp32 chain for the decisions the bound leaves
open) against the oracle's fp32 chain, through the C ABI.

The first layer's levels are decided on the fp32 fmaf chain over (c, ky, kx)
(the oracle's conv2d_f32_seq); the tensor-core path must give the same levels
bit for bit on every output: on the CIFAR and ResNet-stem shapes, ragged
tiles, quantized and fp32 weights, on inputs whose accumulators sit exactly
on a breakpoint or next to one (the exact recompute decides those), and on
pixels with magnitudes the fp16 pieces cannot hold.  The CUDA-core kernel
(plan option first_tensor_cores = 0) gives the same levels."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, convnet_input, convnet_params  # noqa: E402
from tests._gpu import dev_tensor, planes_view  # noqa: E402

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


@pytest.fixture
def restore(M):
    yield
    M.set_plan_options()
    M.minw_test_stall_next_launch(0)


def _gpu_planes(dev, M, x, w, stride, pad, scale, shift, bits_out, bits_w=None, cs=None, tc=True):
    B, C, H, W = x.shape
    O_, _, kh, kw = w.shape
    Ho, Wo = (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1
    M.set_plan_options(first_tensor_cores=int(tc))
    planes = torch.full((M.packed_words(B, O_, Ho, Wo, bits_out),), -1, dtype=torch.int32, device=dev)
    kw_ = {}
    if bits_w:
        kw_["q_w"] = M.quant(bits_w, DEFAULT_THR[bits_w])
        if cs is not None:
            kw_["channel_scale"] = dev_tensor(cs, dev)
    M.minw_conv_first(dev_tensor(x, dev), dev_tensor(w, dev), stride, pad, dev_tensor(scale, dev),
                      dev_tensor(shift, dev), q_out=M.quant(bits_out, DEFAULT_THR[bits_out]), planes_out=planes, **kw_)
    assert M.minw_get_last_device_error() == M.MINW_OK
    return planes_view(planes, B, Ho, Wo, bits_out, O_)


def _ref_planes(x, wl, stride, pad, scale, shift, bits_out):
    y = O.hardtanh(O.affine(O.conv2d_f32_seq(x, wl, stride, pad), scale, shift))
    return O.pack(O.quantize(y, bits_out, DEFAULT_THR[bits_out]), bits_out)


def _levels_w(w, bits_w, cs):
    return O.quantize(w, bits_w, DEFAULT_THR[bits_w], cs).astype(np.float32) if bits_w else w


def _bn(r, O_, K):
    scale = (r.normal(1, 0.1, O_) / np.sqrt(K / 3.0)).astype(np.float32)
    scale[::5] *= -1.0                                   # sigma = -1 channels
    shift = r.normal(0, 0.1, O_).astype(np.float32)
    return scale, shift


CASES = [
    # B, C, H, W, O, k, stride, pad, bits_w (0: fp32 weights), input
    (4, 3, 32, 32, 128, 3, 1, 1, 1, "uniform"),          # CIFAR first layer
    (2, 3, 64, 64, 64, 7, 2, 3, 0, "normal"),            # ResNet stem, fp32 weights
    (2, 3, 64, 64, 64, 7, 2, 3, 3, "normal"),            # stem, 3-bit weights
    (2, 3, 23, 24, 64, 7, 2, 3, 0, "normal"),            # ragged: 12 x 12 outputs, two tiles per image
    (3, 4, 18, 20, 256, 3, 1, 1, 2, "uniform"),          # K = 36 (64-tap blocks), 256 channels
    (2, 8, 17, 16, 192, 3, 2, 1, 0, "normal"),           # K = 72 (two blocks), fp32 weights, stride 2
]


@pytest.mark.parametrize("bits_out", [1, 2, 3])
@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c[:8])) + f"_w{c[8]}_{c[9]}")
def test_first_tc_levels(dev, M, restore, case, bits_out):
    B, C, H, W, O_, k, s, pad, bw, dist = case
    r = np.random.default_rng(B * 100 + C * 10 + bits_out + bw)
    x = (r.uniform(-1, 1, (B, C, H, W)) if dist == "uniform" else r.standard_normal((B, C, H, W))).astype(np.float32)
    w = r.normal(0, 0.05, (O_, C, k, k)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32) if bw > 1 else None
    scale, shift = _bn(r, O_, C * k * k)
    ref = _ref_planes(x, _levels_w(w, bw, cs), s, pad, scale, shift, bits_out)
    got = _gpu_planes(dev, M, x, w, s, pad, scale, shift, bits_out, bw, cs, tc=True)
    assert np.array_equal(got, ref)
    assert np.array_equal(_gpu_planes(dev, M, x, w, s, pad, scale, shift, bits_out, bw, cs, tc=False), ref)


@pytest.mark.parametrize("sign", [1.0, -1.0])
def test_first_tc_exact_ties(dev, M, restore, sign):
    """Inputs on the 2^-6 grid and +-1 weights: every accumulator is an exact
    small multiple of 2^-6 and a breakpoint at 0 or 2^-6 sits exactly on
    thousands of them; the tensor cores cannot settle those decisions and
    the exact chain takes them."""
    B, C, H, W, O_ = 4, 3, 32, 32, 128
    r = np.random.default_rng(5)
    x = (np.round(r.uniform(-1, 1, (B, C, H, W)) * 64) / 64).astype(np.float32)
    w = np.where(r.random((O_, C, 3, 3)) < 0.5, -1.0, 1.0).astype(np.float32)
    scale = np.full(O_, sign, np.float32)
    shift = np.where(np.arange(O_) % 2 == 0, 0.0, sign / 64.0).astype(np.float32)
    for bits_out in (1, 2):
        ref = _ref_planes(x, w, 1, 1, scale, shift, bits_out)
        got = _gpu_planes(dev, M, x, w, 1, 1, scale, shift, bits_out, bits_w=1)
        assert np.array_equal(got, ref)


def test_first_tc_near_ties(dev, M, restore):
    """Random fp32 inputs with each channel's breakpoint placed on the chain
    value of one of its outputs (and one ulp off it): the decisions there
    hinge on the last bit of the fp32 chain."""
    B, C, H, W, O_ = 2, 3, 64, 64, 64
    r = np.random.default_rng(11)
    x = r.standard_normal((B, C, H, W)).astype(np.float32)
    w = r.normal(0, 0.05, (O_, C, 7, 7)).astype(np.float32)
    acc = O.conv2d_f32_seq(x, w, 2, 3)
    scale = np.ones(O_, np.float32)
    pick = acc[r.integers(0, B, O_), np.arange(O_), r.integers(0, 32, O_), r.integers(0, 32, O_)]
    shift = (-pick).astype(np.float32)
    shift[1::3] = np.nextafter(shift[1::3], np.float32(np.inf))
    shift[2::3] = np.nextafter(shift[2::3], np.float32(-np.inf))
    ref = _ref_planes(x, w, 2, 3, scale, shift, 1)
    got = _gpu_planes(dev, M, x, w, 2, 3, scale, shift, 1)
    assert np.array_equal(got, ref)


def test_first_tc_large_pixels(dev, M, restore):
    """Pixels with inputs beyond the fp16 pieces' range (|x| >= 2^15, and
    above the fp16 maximum) are recomputed on the fp32 chain as a whole."""
    B, C, H, W, O_ = 2, 3, 32, 32, 128
    r = np.random.default_rng(12)
    x = r.uniform(-1, 1, (B, C, H, W)).astype(np.float32)
    x[0, 0, 3, 4] = 5.0e4
    x[0, 2, 10, 10] = -7.0e4
    x[1, 1, 31, 31] = 3.0e4
    x[1, 0, 0, 0] = 1.0e30
    w = r.normal(0, 0.05, (O_, C, 3, 3)).astype(np.float32)
    scale, shift = _bn(r, O_, 27)
    for bw in (0, 1):
        ref = _ref_planes(x, _levels_w(w, bw, None), 1, 1, scale, shift, 2)
        got = _gpu_planes(dev, M, x, w, 1, 1, scale, shift, 2, bw)
        assert np.array_equal(got, ref)


def test_first_tc_timeout(dev, M, restore):
    """The tensor-core first layer with a stalled MMA issuer: MINW_ETIMEOUT
    once, the kernel winds down (patches drained, TMEM freed), then a correct
    run and MINW_OK."""
    assert M.minw_get_last_device_error() == M.MINW_OK
    r = np.random.default_rng(13)
    x = r.uniform(-1, 1, (3, 3, 16, 16)).astype(np.float32)
    w = r.normal(0, 0.05, (64, 3, 3, 3)).astype(np.float32)
    sc, sh = _bn(r, 64, 27)
    xd, wd, scd, shd = (dev_tensor(a, dev) for a in (x, w, sc, sh))
    planes = torch.empty(M.packed_words(3, 64, 16, 16, 1), dtype=torch.int32, device=dev)
    M.set_plan_options(wait_cycles=1 << 20)
    M.minw_test_stall_next_launch(M.STALL_CONV_FIRST)
    M.minw_conv_first(xd, wd, 1, 1, scd, shd, q_w=M.quant(1, DEFAULT_THR[1]), q_out=M.quant(1, DEFAULT_THR[1]),
                      planes_out=planes)
    assert M.minw_get_last_device_error() == M.MINW_ETIMEOUT
    M.minw_conv_first(xd, wd, 1, 1, scd, shd, q_w=M.quant(1, DEFAULT_THR[1]), q_out=M.quant(1, DEFAULT_THR[1]),
                      planes_out=planes)
    assert M.minw_get_last_device_error() == M.MINW_OK
    ref = _ref_planes(x, O.quantize(w, 1, DEFAULT_THR[1]), 1, 1, sc, sh, 1)
    assert np.array_equal(planes_view(planes, 3, 16, 16, 1, 64), ref)


@pytest.mark.parametrize("tc", [0, 1])
def test_convnet_first_layer_paths(dev, M, restore, tc):
    """The CIFAR ConvNet (E2M1 codes out of the first layer) with either
    first-layer kernel: logits equal to the oracle's."""
    M.set_plan_options(first_tensor_cores=tc)
    p = convnet_params(21, bits_a=1, bits_w=1)
    x = convnet_input(22, 6)
    net = M.Net(M.layer_descs(p, dev), max_batch=6)
    logits = torch.empty((6, 10), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    assert M.minw_get_last_device_error() == M.MINW_OK
    assert np.array_equal(logits.cpu().numpy(), N.convnet_forward(p, x))
    net.close()
