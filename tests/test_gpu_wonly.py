"""GPU parity of the weight-only quantized convolution (full-precision bf16
activations times 1-3-bit weights on the tcgen05 tensor cores, kind::f16)
against the oracle, through the C ABI: the bf16 NHWC conversion and the bf16
level weights bit for bit, and the convolution within the bound of fp32
accumulation (the tensor core's summation order is its own):
|y - y_ref| <= |scale| K 2^-23 A + 2^-23 |y_ref|, with A = sum |x w| of the
output, which covers rounding or truncating additions; a wrong product, tap
or channel breaks it by orders of magnitude."""
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


def _operands(dev, M, x, w, bits, cs):
    B, C, H, W = x.shape
    O_, _, kh, kw = w.shape
    xb = torch.empty((B, H, W, C), dtype=torch.int16, device=dev)
    wb = torch.empty((O_, kh, kw, C), dtype=torch.int16, device=dev)
    M.minw_to_bf16_nhwc(dev_tensor(x, dev), xb)
    M.minw_pack_weight_bf16(dev_tensor(w, dev), M.quant(bits, DEFAULT_THR[bits]), wb,
                            channel_scale=dev_tensor(cs, dev))
    return xb, wb


def _bf16_values(t):
    """int16 bit patterns of bf16 -> fp32 values (upper half of the word)."""
    u = t.cpu().numpy().view(np.uint16).astype(np.uint32) << 16
    return u.view(np.float32)


@pytest.mark.parametrize("shape", [(2, 64, 5, 7), (1, 128, 3, 9), (3, 96, 4, 4)])
def test_to_bf16_nhwc(dev, M, shape):
    x = (np.random.default_rng(sum(shape)).standard_normal(shape) * 3).astype(np.float32)
    B, C, H, W = shape
    out = torch.empty((B, H, W, C), dtype=torch.int16, device=dev)
    M.minw_to_bf16_nhwc(dev_tensor(x, dev), out)
    want = O.bf16_round(x).transpose(0, 2, 3, 1)
    assert np.array_equal(_bf16_values(out).view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_pack_weight_bf16(dev, M, bits):
    w = np.random.default_rng(bits).normal(0, 0.05, (24, 64, 3, 3)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(24, -1)).max(1)).astype(np.float32)
    out = torch.empty((24, 3, 3, 64), dtype=torch.int16, device=dev)
    M.minw_pack_weight_bf16(dev_tensor(w, dev), M.quant(bits, DEFAULT_THR[bits]), out,
                            channel_scale=dev_tensor(cs, dev))
    units = O.quantize(w, bits, DEFAULT_THR[bits], cs) * 2.0 ** O.units_shift(bits)
    assert np.array_equal(_bf16_values(out).astype(np.float64), units.transpose(0, 2, 3, 1))


CASES = [(2, 64, 10, 12, 96, 1, 0), (3, 128, 9, 9, 128, 2, 0), (2, 256, 8, 8, 256, 1, 1), (1, 64, 7, 7, 320, 1, 0)]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("bits", [1, 2, 3])
def test_conv2d_bf16(dev, M, case, bits):
    B, C, H, W, O_, s, pool = case
    r = np.random.default_rng(1000 * bits + sum(case))
    x = r.standard_normal((B, C, H, W)).astype(np.float32)
    w = r.normal(0, 0.05, (O_, C, 3, 3)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32)
    scale = r.normal(0.01, 0.005, O_).astype(np.float32)
    shift = r.normal(0, 0.1, O_).astype(np.float32)
    xb, wb = _operands(dev, M, x, w, bits, cs)
    Ho, Wo = (H - 1) // s + 1, (W - 1) // s + 1
    Hp, Wp = (Ho // 2, Wo // 2) if pool else (Ho, Wo)
    y = torch.full((B, O_, Hp, Wp), np.nan, dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(xb, B, C, H, W, wb, O_, 3, 3, bits, s, 1, pool, dev_tensor(scale, dev),
                       dev_tensor(shift, dev), y)
    torch.cuda.synchronize()
    xr = O.bf16_round(x).astype(np.float64)
    wu = O.quantize(w, bits, DEFAULT_THR[bits], cs) * 2.0 ** O.units_shift(bits)
    acc = O.conv2d_real(xr, wu, s, 1)
    A = O.conv2d_real(np.abs(xr), np.abs(wu), s, 1)
    if pool:
        acc, A = O.maxpool_f64(acc), O.maxpool_f64(A)
    sc = scale.astype(np.float64)[None, :, None, None]
    yref = acc * sc + shift.astype(np.float64)[None, :, None, None]
    K = C * 9
    bound = np.abs(sc) * K * 2.0 ** -23 * A + 2.0 ** -23 * np.abs(yref) + 1e-30
    err = np.abs(y.cpu().numpy().astype(np.float64) - yref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound)}"


def test_conv2d_bf16_sweep_shape_sampled(dev, M):
    """The bit-width sweep's shape, 256 x 512 x 14 x 14 -> 512 (3x3, K = 4608),
    with 1-bit weights: images 0 and 255 against the oracle."""
    B, C, H, W, O_ = 256, 512, 14, 14, 512
    r = np.random.default_rng(77)
    x = r.standard_normal((B, C, H, W)).astype(np.float32)
    w = r.standard_normal((O_, C, 3, 3)).astype(np.float32)
    cs = np.ones(O_, dtype=np.float32)
    scale = np.full(O_, 1.0 / 64, dtype=np.float32)
    shift = np.zeros(O_, dtype=np.float32)
    xb, wb = _operands(dev, M, x, w, 1, cs)
    y = torch.empty((B, O_, H, W), dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(xb, B, C, H, W, wb, O_, 3, 3, 1, 1, 1, 0, dev_tensor(scale, dev), dev_tensor(shift, dev), y)
    torch.cuda.synchronize()
    pick = [0, B - 1]
    xr = O.bf16_round(x[pick]).astype(np.float64)
    wu = O.quantize(w, 1, DEFAULT_THR[1])
    acc = O.conv2d_real(xr, wu, 1, 1)
    A = O.conv2d_real(np.abs(xr), np.abs(wu), 1, 1)
    yref = acc / 64.0
    bound = (1.0 / 64) * C * 9 * 2.0 ** -23 * A + 2.0 ** -23 * np.abs(yref) + 1e-30
    err = np.abs(y.cpu().numpy()[pick].astype(np.float64) - yref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound)}"


@pytest.mark.parametrize("B,K,O_", [(256, 1152, 256), (200, 2048, 512)])
def test_conv2d_bf16_fully_connected_cta_pairs(dev, M, B, K, O_):
    """A fully connected shape long enough for CTA pairs (K / 64 >= 18 bf16 K
    blocks, O a multiple of 256, no workspace): the pair kernel with the
    row-contiguous staged stores of 1 x 1 outputs, against the oracle within
    the fp32 accumulation bound; B = 200 leaves a ragged, odd pixel tile."""
    r = np.random.default_rng(B + K + O_)
    x = r.standard_normal((B, K, 1, 1)).astype(np.float32)
    w = r.normal(0, 0.05, (O_, K, 1, 1)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32)
    scale = r.normal(0.01, 0.005, O_).astype(np.float32)
    shift = r.normal(0, 0.1, O_).astype(np.float32)
    xb, wb = _operands(dev, M, x, w, 1, cs)
    y = torch.full((B, O_, 1, 1), np.nan, dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(xb, B, K, 1, 1, wb, O_, 1, 1, 1, 1, 0, 0, dev_tensor(scale, dev), dev_tensor(shift, dev), y)
    torch.cuda.synchronize()
    xr = O.bf16_round(x).reshape(B, K).astype(np.float64)
    wu = O.quantize(w, 1, DEFAULT_THR[1], cs).reshape(O_, K).astype(np.float64)
    acc, A = xr @ wu.T, np.abs(xr) @ np.abs(wu).T
    yref = acc * scale.astype(np.float64) + shift.astype(np.float64)
    bound = np.abs(scale.astype(np.float64)) * K * 2.0 ** -23 * A + 2.0 ** -23 * np.abs(yref) + 1e-30
    err = np.abs(y.cpu().numpy().reshape(B, O_).astype(np.float64) - yref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound)}"
    assert M.minw_get_last_device_error() == M.MINW_OK


def test_conv2d_bf16_errors(dev, M):
    xb = torch.zeros((1, 4, 4, 32), dtype=torch.int16, device=dev)
    wb = torch.zeros((8, 3, 3, 32), dtype=torch.int16, device=dev)
    sc = torch.ones(8, device=dev)
    y = torch.empty((1, 8, 4, 4), device=dev)
    with pytest.raises(M.MinwError):
        M.minw_conv2d_bf16(xb, 1, 32, 4, 4, wb, 8, 3, 3, 1, 1, 1, 0, sc, sc, y)     # C % 64 != 0
    with pytest.raises(M.MinwError):
        M.minw_conv2d_bf16(xb, 1, 32, 4, 4, wb, 8, 3, 3, 1, 1, 1, 0, sc, sc, None)  # no output


# Narrow layers of the Table III networks (3-bit weights, full-precision activations):
# B, C, H, W, O, k, stride, pad
NARROW = [
    (4, 16, 32, 32, 16, 3, 1, 1),     # ResNet-110 stage 1 (16 channels at 32 x 32)
    (4, 16, 32, 32, 32, 3, 2, 1),     # ResNet-110 entering stage 2 (stride 2)
    (4, 16, 32, 32, 32, 1, 2, 0),     # its 1 x 1 / 2 shortcut
    (4, 32, 16, 16, 32, 3, 1, 1),     # ResNet-110 stage 2
    (4, 48, 32, 32, 48, 1, 1, 0),     # DenseNet-BC-100 bottleneck (24 + 2 x 12 channels in, 4 x 12 out)
    (4, 48, 32, 32, 12, 3, 1, 1),     # DenseNet-BC-100 3 x 3, growth 12
    (4, 96, 16, 16, 48, 1, 1, 0),     # DenseNet-BC-100 transition (compression 1/2)
]


@pytest.mark.parametrize("case", NARROW)
def test_conv2d_bf16_narrow_channels(dev, M, case):
    """Channel counts that are not a multiple of 64 run on zero-padded
    operands (minw_to_bf16_nhwc_pad, minw_pack_weight_bf16_pad; a zero adds
    exactly 0 to every product): the padded conversions bit for bit, and the
    convolution of the padded operands within the fp32-accumulation bound of
    the oracle's product of the unpadded ones, 3-bit weights."""
    B, C, H, W, O_, k, s, pad = case
    bits = 3
    Cp = (C + 63) // 64 * 64
    r = np.random.default_rng(sum(case) * 7 + 3)
    x = r.standard_normal((B, C, H, W)).astype(np.float32)
    w = r.normal(0, 0.05, (O_, C, k, k)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32)
    scale = r.normal(0.01, 0.005, O_).astype(np.float32)
    shift = r.normal(0, 0.1, O_).astype(np.float32)
    xb = torch.full((B, H, W, Cp), 0x7FFF, dtype=torch.int16, device=dev)       # stale contents: overwritten
    wb = torch.full((O_, k, k, Cp), 0x7FFF, dtype=torch.int16, device=dev)
    M.minw_to_bf16_nhwc_pad(dev_tensor(x, dev), Cp, xb)
    M.minw_pack_weight_bf16_pad(dev_tensor(w, dev), Cp, M.quant(bits, DEFAULT_THR[bits]), wb,
                                channel_scale=dev_tensor(cs, dev))
    xr = O.bf16_round(x)
    wu = O.quantize(w, bits, DEFAULT_THR[bits], cs) * 2.0 ** O.units_shift(bits)
    xv, wv = _bf16_values(xb), _bf16_values(wb)
    assert np.array_equal(xv[..., :C].view(np.uint32), xr.transpose(0, 2, 3, 1).view(np.uint32))
    assert not xv[..., C:].view(np.uint32).any()
    assert np.array_equal(wv[..., :C].astype(np.float64), wu.transpose(0, 2, 3, 1))
    assert not wv[..., C:].view(np.uint32).any()
    Ho, Wo = (H + 2 * pad - k) // s + 1, (W + 2 * pad - k) // s + 1
    y = torch.full((B, O_, Ho, Wo), np.nan, dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(xb, B, Cp, H, W, wb, O_, k, k, bits, s, pad, 0, dev_tensor(scale, dev),
                       dev_tensor(shift, dev), y)
    torch.cuda.synchronize()
    xr64 = xr.astype(np.float64)
    acc = O.conv2d_real(xr64, wu, s, pad)
    A = O.conv2d_real(np.abs(xr64), np.abs(wu), s, pad)
    sc = scale.astype(np.float64)[None, :, None, None]
    yref = acc * sc + shift.astype(np.float64)[None, :, None, None]
    K = Cp * k * k
    bound = np.abs(sc) * K * 2.0 ** -23 * A + 2.0 ** -23 * np.abs(yref) + 1e-30
    err = np.abs(y.cpu().numpy().astype(np.float64) - yref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound)}"


# B, C, ldc, H, W, O, k, stride, out_ld, out_off
HT_CASES = [
    (4, 64, 256, 32, 32, 48, 1, 1, 64, 0),      # DenseNet-100 bottleneck: the first 64 of 256-element rows
    (4, 64, 0, 32, 32, 12, 3, 1, 256, 36),      # DenseNet-100 3x3 appending 12 channels at 36 (8-byte aligned)
    (3, 64, 0, 16, 16, 12, 3, 1, 320, 110),     # ... at 110 (4-byte aligned)
    (2, 128, 0, 8, 8, 32, 3, 2, 64, 0),         # stride 2, 16-byte aligned rows
    (2, 64, 128, 9, 7, 40, 3, 1, 48, 5),        # ragged tiles, odd offset
]


@pytest.mark.parametrize("case,residual", [(c, False) for c in HT_CASES] + [(HT_CASES[3], True), (HT_CASES[4], True)])
def test_conv2d_bf16_hardtanh(dev, M, case, residual):
    """The fused HardTanh + bf16 NHWC epilogue equals the bf16 rounding of
    HardTanh of minw_conv2d_bf16's output [plus a shortcut, one fp32 add] on
    the same operands bit for bit (the same accumulators), lands in channels
    out_off .. out_off + O of each out_ld-element row and writes nothing
    else, and its fp32 NCHW copy equals the clamped value; inputs read from
    the first C elements of ldc-element rows whose other elements hold values
    far out of range (a read of them would show)."""
    B, C, ldc, H, W, O_, k, s, ld, off = case
    pad = k // 2
    r = np.random.default_rng(sum(case) * 5 + 1)
    Cf = ldc or C
    x = r.standard_normal((B, Cf, H, W)).astype(np.float32)
    x[:, C:] = 1e30
    w = r.normal(0, 0.05, (O_, C, k, k)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(O_, -1)).max(1)).astype(np.float32)
    scale = r.normal(0.02, 0.01, O_).astype(np.float32)
    shift = r.normal(0, 0.3, O_).astype(np.float32)
    bits = 3
    xw = torch.empty((B, H, W, Cf), dtype=torch.int16, device=dev)
    M.minw_to_bf16_nhwc(dev_tensor(x, dev), xw)
    xc, wb = _operands(dev, M, np.ascontiguousarray(x[:, :C]), w, bits, cs)
    Ho, Wo = (H + 2 * pad - k) // s + 1, (W + 2 * pad - k) // s + 1
    sc, sh = dev_tensor(scale, dev), dev_tensor(shift, dev)
    y = torch.empty((B, O_, Ho, Wo), dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(xc, B, C, H, W, wb, O_, k, k, bits, s, pad, 0, sc, sh, y)
    sentinel = 0x7F7F
    out = torch.full((B, Ho, Wo, ld), sentinel, dtype=torch.int16, device=dev)
    res = r.uniform(-1, 1, (B, O_, Ho, Wo)).astype(np.float32) if residual else None
    z = torch.full((B, O_, Ho, Wo), np.nan, dtype=torch.float32, device=dev) if residual else None
    M.minw_conv2d_bf16_hardtanh(xw, B, C, H, W, ldc, wb, O_, k, k, bits, s, pad, sc, sh, out, ld, off,
                                residual=dev_tensor(res, dev) if residual else None, y_out=z)
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint16)
    v = y.cpu().numpy()
    if residual:
        v = (v + res).astype(np.float32)
    v = np.clip(v, -1.0, 1.0)
    if residual:
        assert np.array_equal(z.cpu().numpy(), v)
    want = O.bf16_round(v).transpose(0, 2, 3, 1)
    want_bits = (want.view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal(got[..., off:off + O_], want_bits)
    rest = np.concatenate([got[..., :off].ravel(), got[..., off + O_:].ravel()])
    assert (rest == sentinel).all()
    assert M.minw_get_last_device_error() == M.MINW_OK


def test_conv2d_bf16_hardtanh_errors(dev, M):
    xb = torch.zeros((1, 4, 4, 64), dtype=torch.int16, device=dev)
    wb = torch.zeros((8, 1, 1, 64), dtype=torch.int16, device=dev)
    sc = torch.ones(8, device=dev)
    out = torch.zeros((1, 4, 4, 16), dtype=torch.int16, device=dev)
    with pytest.raises(M.MinwError):       # the row cannot hold channels 10 .. 18
        M.minw_conv2d_bf16_hardtanh(xb, 1, 64, 4, 4, 0, wb, 8, 1, 1, 1, 1, 0, sc, sc, out, 16, 10)
    with pytest.raises(M.MinwError):       # input rows shorter than C
        M.minw_conv2d_bf16_hardtanh(xb, 1, 64, 4, 4, 32, wb, 8, 1, 1, 1, 1, 0, sc, sc, out, 16, 0)
