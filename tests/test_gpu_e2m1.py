"""GPU parity of the E2M1 operand path (FP4 level codes, two channels per
byte, tcgen05 kind::mxf4 with unit block scales) against the oracle, through
the C ABI: the code layout, exact accumulators for all nine bit-width pairs
on ragged tiles, strided and CTA-pair shapes and at the largest magnitudes,
the fused block epilogue writing E2M1 codes (pixel-major and channel-major
tiles, pooled), a residual shortcut held as E2M1 codes, and whole networks
whose hidden layers run on E2M1 operands."""
from itertools import product

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem, convnet_input, convnet_params  # noqa: E402
from tests._gpu import case_seed, dev_tensor, planes_view  # noqa: E402

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


def decode_e2m1(b, C):
    """E2M1 bytes [..., C / 2] to values [..., C] from the format's definition
    (1 sign bit, 2 exponent bits with bias 1, 1 mantissa bit; exponent 0 is
    the subnormal range): channel 2j in the low nibble of byte j."""
    b = np.asarray(b).astype(np.int64)
    nib = np.stack([b & 0xF, b >> 4], axis=-1).reshape(b.shape[:-1] + (C,))
    sign = np.where(nib & 8, -1.0, 1.0)
    e = (nib >> 1) & 3
    m = nib & 1
    mag = np.where(e == 0, m * 0.5, (1.0 + m / 2.0) * np.power(2.0, e - 1.0))
    return sign * mag


@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("shape", [(2, 128, 5, 7), (1, 64, 3, 3), (3, 32, 1, 1)])
def test_quantize_codes_e2m1(dev, M, bits, shape):
    B, C, H, W = shape
    x = np.random.default_rng(C + bits + 7).standard_normal(shape).astype(np.float32)
    codes = torch.empty((B, H, W, C // 2), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes_e2m1(dev_tensor(x, dev), M.quant(bits, DEFAULT_THR[bits]), codes)
    lv = O.quantize(x, bits, DEFAULT_THR[bits]) * 2.0 ** O.units_shift(bits)
    assert np.array_equal(decode_e2m1(codes.cpu().numpy(), C), lv.transpose(0, 2, 3, 1))


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_weight_codes_e2m1(dev, M, bits):
    w = np.random.default_rng(bits + 40).normal(0, 0.05, (40, 256, 3, 3)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(40, -1)).max(1)).astype(np.float32)
    codes = torch.empty((40, 3, 3, 128), dtype=torch.uint8, device=dev)
    M.minw_pack_weight_codes_e2m1(dev_tensor(w, dev), M.quant(bits, DEFAULT_THR[bits]), codes,
                                  channel_scale=dev_tensor(cs, dev))
    lv = O.quantize(w, bits, DEFAULT_THR[bits], cs) * 2.0 ** O.units_shift(bits)
    assert np.array_equal(decode_e2m1(codes.cpu().numpy(), 256), lv.transpose(0, 2, 3, 1))


def _operands(dev, M, p):
    B, C, H, W, O_ = p["B"], p["C"], p["H"], p["W"], p["O"]
    act = torch.empty((B, H, W, C // 2), dtype=torch.uint8, device=dev)
    wgt = torch.empty((O_, p["kh"], p["kw"], C // 2), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes_e2m1(dev_tensor(p["x"], dev), M.quant(p["bits_a"], p["thr_a"]), act)
    M.minw_pack_weight_codes_e2m1(dev_tensor(p["w"], dev), M.quant(p["bits_w"], p["thr_w"]), wgt,
                                  channel_scale=dev_tensor(p["w_scale"], dev))
    return act, wgt


def _ref_acc(p):
    al = O.quantize(p["x"], p["bits_a"], p["thr_a"])
    wl = O.quantize(p["w"], p["bits_w"], p["thr_w"], p["w_scale"])
    return O.conv2d_levels(al, wl, p["stride"], p["pad"], p["bits_a"], p["bits_w"])


def _out_hw(p):
    return ((p["H"] + 2 * p["pad"] - p["kh"]) // p["stride"] + 1,
            (p["W"] + 2 * p["pad"] - p["kw"]) // p["stride"] + 1)


CASES = [
    # B, C, H, W, O, k, stride, pad
    (2, 128, 9, 7, 70, 3, 1, 1),      # ragged pixel tile and channel tile (two accumulators)
    (3, 256, 16, 16, 256, 3, 1, 1),   # 256-channel tile (one accumulator), 128-byte rows
    (2, 128, 8, 8, 10, 1, 1, 0),      # O = 10: one 16-wide channel tile
    (130, 512, 4, 4, 20, 4, 1, 0),    # fully connected over a 4x4 map, two image tiles
    (2, 128, 1, 1, 300, 1, 1, 0),     # two channel tiles, the second ragged
    (1, 128, 14, 14, 64, 3, 1, 1),    # 14x14: tiles overhang both edges
    (2, 256, 16, 16, 128, 3, 2, 1),   # stride 2
    (3, 512, 8, 8, 512, 3, 1, 1),     # 18 K blocks, 256-channel tiles: CTA pairs, odd pixel-tile count
]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("ba,bw", list(product([1, 2, 3], [1, 2, 3])))
def test_conv_e2m1(dev, M, case, ba, bw):
    B, C, H, W, O_, k, stride, pad = case
    p = conv_problem(case_seed(case, ba, bw, "e2m1"), B, C, H, W, O_, k, k, stride, pad, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    Ho, Wo = _out_hw(p)
    acc = torch.full((B, O_, Ho, Wo), -7, dtype=torch.int32, device=dev)
    y = torch.empty(acc.shape, dtype=torch.float32, device=dev)
    M.minw_conv_block_codes_ex(act, B, C, H, W, ba, wgt, O_, k, k, bw, stride, pad, 0,
                               dev_tensor(p["scale"], dev), dev_tensor(p["shift"], dev), y_out=y,
                               in_format=M.CODES_E2M1, acc_out=acc)
    ref = _ref_acc(p)
    got = acc.cpu().numpy()
    assert np.array_equal(got, ref), f"{np.sum(got != ref)} of {ref.size} accumulators differ"
    assert np.array_equal(y.cpu().numpy(), O.affine(ref, p["scale"], p["shift"]))
    assert M.minw_get_last_device_error() == M.MINW_OK


PAIR_CASES = [
    # B, C, H, W, O, k, stride, pad
    (3, 512, 8, 8, 512, 3, 1, 1),     # odd pixel-tile count: the last pair holds one padded tile
    (2, 256, 14, 14, 384, 3, 1, 1),   # 14x14 tiles overhang both edges, three 128-channel tiles
    (4, 128, 16, 16, 128, 3, 2, 1),   # stride 2, one channel tile
    (2, 128, 8, 8, 96, 3, 1, 1),      # O % 128 != 0: the request falls back to the default tiling
]


@pytest.mark.parametrize("case", PAIR_CASES)
@pytest.mark.parametrize("ba,bw", [(1, 1), (2, 3), (3, 3)])
def test_conv_e2m1_pairs_single_layer(dev, M, case, ba, bw):
    """A single E2M1 convolution asked to run as CTA pairs of 256 pixels x
    128 channels (minw_block_extra.e2m1_pairs): the same exact accumulators as
    the oracle's, wherever the shape allows the pairs and where it does not."""
    B, C, H, W, O_, k, stride, pad = case
    seed = (7 * B + C + 3 * O_ + 5 * H + 11 * ba + 13 * bw) % 1000
    p = conv_problem(seed, B, C, H, W, O_, k, k, stride, pad, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    Ho, Wo = _out_hw(p)
    acc = torch.full((B, O_, Ho, Wo), -7, dtype=torch.int32, device=dev)
    M.minw_conv_block_codes_ex(act, B, C, H, W, ba, wgt, O_, k, k, bw, stride, pad, 0, None, None,
                               in_format=M.CODES_E2M1, acc_out=acc, e2m1_pairs=True)
    ref = _ref_acc(p)
    got = acc.cpu().numpy()
    assert np.array_equal(got, ref), f"{np.sum(got != ref)} of {ref.size} accumulators differ"
    assert M.minw_get_last_device_error() == M.MINW_OK


@pytest.mark.parametrize("ba,bw,hw,O_", [(1, 1, 32, 96), (2, 2, 16, 256), (3, 3, 8, 96), (2, 1, 16, 160)])
def test_block_e2m1_pool(dev, M, ba, bw, hw, O_):
    """Pooled block whose quantized output goes out as E2M1 codes and planes,
    with the fp32 BN output beside them."""
    B, C = 2, 128
    p = conv_problem(71 + ba + 3 * bw + hw, B, C, hw, hw, O_, 3, 3, 1, 1, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    bo = ba
    h2 = hw // 2
    codes = torch.full((B, h2, h2, O_ // 2), 0x77, dtype=torch.uint8, device=dev)
    planes = torch.full((M.packed_words(B, O_, h2, h2, bo),), -1, dtype=torch.int32, device=dev)
    y = torch.empty((B, O_, h2, h2), dtype=torch.float32, device=dev)
    M.minw_conv_block_codes_ex(act, B, C, hw, hw, ba, wgt, O_, 3, 3, bw, 1, 1, 1, dev_tensor(p["scale"], dev),
                               dev_tensor(p["shift"], dev), q_out=M.quant(bo, DEFAULT_THR[bo]), codes_out=codes,
                               planes_out=planes, y_out=y, in_format=M.CODES_E2M1, out_format=M.CODES_E2M1)
    acc = O.maxpool_i32(_ref_acc(p), 2, 2)
    yr = O.hardtanh(O.affine(acc, p["scale"], p["shift"]))
    assert np.array_equal(y.cpu().numpy(), yr)
    lv = O.quantize(yr, bo, DEFAULT_THR[bo])
    assert np.array_equal(planes_view(planes, B, h2, h2, bo, O_), O.pack(lv, bo))
    assert np.array_equal(decode_e2m1(codes.cpu().numpy(), O_), (lv * 2.0 ** O.units_shift(bo)).transpose(0, 2, 3, 1))


@pytest.mark.parametrize("O_,pool,bits", [(128, 1, 1), (128, 0, 3), (64, 0, 2)])
def test_block_e2m1_channel_major(dev, M, O_, pool, bits):
    """Codes-only outputs of a 64- or 128-channel layer with enough 256-pixel
    tiles run as channel-major tiles (128 channels x 256 pixels); the E2M1
    output codes equal the E4M3 path's (decoded) on the whole batch, and the
    oracle's on the first and last image."""
    B, C, hw = 160, 128, 32
    p = conv_problem(91 + O_ + pool + bits, B, C, hw, hw, O_, 3, 3, 1, 1, bits, bits, w_sigma=0.5)
    act4, wgt4 = _operands(dev, M, p)
    act8 = torch.empty((B, hw, hw, C), dtype=torch.uint8, device=dev)
    wgt8 = torch.empty((O_, 3, 3, C), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(bits, p["thr_a"]), act8)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(bits, p["thr_w"]), wgt8,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    ho = hw // 2 if pool else hw
    q = M.quant(bits, DEFAULT_THR[bits])
    sc, sh = dev_tensor(p["scale"], dev), dev_tensor(p["shift"], dev)
    c4 = torch.full((B, ho, ho, O_ // 2), 0x77, dtype=torch.uint8, device=dev)
    c8 = torch.full((B, ho, ho, O_), 0x77, dtype=torch.uint8, device=dev)
    M.minw_conv_block_codes_ex(act4, B, C, hw, hw, bits, wgt4, O_, 3, 3, bits, 1, 1, pool, sc, sh, q_out=q,
                               codes_out=c4, in_format=M.CODES_E2M1, out_format=M.CODES_E2M1)
    M.minw_conv_block_codes(act8, B, C, hw, hw, bits, wgt8, O_, 3, 3, bits, 1, 1, pool, sc, sh, q_out=q, codes_out=c8)
    torch.cuda.synchronize()
    from tests.test_gpu_tc import decode_e4m3
    v4 = decode_e2m1(c4.cpu().numpy(), O_)
    assert np.array_equal(v4, decode_e4m3(c8.cpu().numpy()))
    for b in (0, B - 1):
        sub = dict(p, x=p["x"][b:b + 1], B=1)
        acc = _ref_acc(sub)
        if pool:
            acc = O.maxpool_i32(acc, 2, 2)
        lv = O.quantize(O.hardtanh(O.affine(acc, p["scale"], p["shift"])), bits, DEFAULT_THR[bits])
        assert np.array_equal(v4[b:b + 1], (lv * 2.0 ** O.units_shift(bits)).transpose(0, 2, 3, 1))
    assert M.minw_get_last_device_error() == M.MINW_OK


@pytest.mark.parametrize("bits", [1, 3])
def test_block_e2m1_residual(dev, M, bits):
    """Residual block: y = BN(acc) + shortcut, the shortcut given as E2M1
    codes of a level tensor, then HardTanh and the quantizer, out as E2M1."""
    B, C, hw, O_ = 2, 128, 8, 128
    p = conv_problem(33 + bits, B, C, hw, hw, O_, 3, 3, 1, 1, bits, bits, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    r = np.random.default_rng(5 + bits).standard_normal((B, O_, hw, hw)).astype(np.float32)
    res = torch.empty((B, hw, hw, O_ // 2), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes_e2m1(dev_tensor(r, dev), M.quant(bits, DEFAULT_THR[bits]), res)
    codes = torch.full((B, hw, hw, O_ // 2), 0x77, dtype=torch.uint8, device=dev)
    M.minw_conv_block_codes_ex(act, B, C, hw, hw, bits, wgt, O_, 3, 3, bits, 1, 1, 0, dev_tensor(p["scale"], dev),
                               dev_tensor(p["shift"], dev), q_out=M.quant(bits, DEFAULT_THR[bits]), codes_out=codes,
                               res_codes=res, res_bits=bits, in_format=M.CODES_E2M1, out_format=M.CODES_E2M1,
                               res_format=M.CODES_E2M1)
    y_bn = O.affine(_ref_acc(p), p["scale"], p["shift"])
    rl = O.quantize(r, bits, DEFAULT_THR[bits])
    yr = O.hardtanh((y_bn + rl.astype(np.float32)).astype(np.float32))
    lv = O.quantize(yr, bits, DEFAULT_THR[bits])
    assert np.array_equal(decode_e2m1(codes.cpu().numpy(), O_), (lv * 2.0 ** O.units_shift(bits)).transpose(0, 2, 3, 1))


def _adversarial(bits, C, k, hw, B=2, O_=64):
    """Image 0 at the largest level everywhere; image 1 at the largest level on
    the first half of the channels and the smallest non-zero level on the
    rest, so unit products follow large partial sums."""
    big, small = 1.0, (0.2 if bits == 3 else 1.0)
    x = np.full((B, C, hw, hw), big, dtype=np.float32)
    x[1, C // 2:] = small
    w = np.full((O_, C, k, k), big, dtype=np.float32)
    if bits == 3:
        w[1::2, ::7] = 0.45
        w[1::2, 3::5] = 0.2
    elif bits == 2:
        w[1::2, ::3] = 0.0
    return dict(x=x, w=w, w_scale=np.ones(O_, np.float32), thr_a=DEFAULT_THR[bits], thr_w=DEFAULT_THR[bits],
                scale=np.ones(O_, np.float32), shift=np.zeros(O_, np.float32), B=B, C=C, H=hw, W=hw, O=O_,
                kh=k, kw=k, stride=1, pad=(k - 1) // 2 if k == 3 else 0, bits_a=bits, bits_w=bits)


@pytest.mark.parametrize("bits,C,k,hw", [(3, 512, 3, 6), (1, 512, 4, 4), (1, 1024, 1, 1), (2, 512, 3, 5)])
def test_e2m1_exact_at_largest_magnitudes(dev, M, bits, C, k, hw):
    """|acc| up to 16 * 4608 with unit products next to the largest: the
    block-scaled FP4 contraction reproduces every integer exactly."""
    p = _adversarial(bits, C, k, hw)
    act, wgt = _operands(dev, M, p)
    Ho, Wo = _out_hw(p)
    acc = torch.empty((p["B"], p["O"], Ho, Wo), dtype=torch.int32, device=dev)
    M.minw_conv_block_codes_ex(act, p["B"], C, hw, hw, bits, wgt, p["O"], k, k, bits, 1, p["pad"], 0,
                               None, None, in_format=M.CODES_E2M1, acc_out=acc)
    ref = _ref_acc(p)
    assert np.abs(ref).max() == (16 if bits == 3 else 1) * C * k * k
    assert np.array_equal(acc.cpu().numpy(), ref)


def test_e2m1_unsupported_channels(dev, M):
    """E2M1 operands need 64-byte rows: C = 64 is refused before any launch."""
    act = torch.zeros((1, 8, 8, 32), dtype=torch.uint8, device=dev)
    wgt = torch.zeros((64, 3, 3, 32), dtype=torch.uint8, device=dev)
    acc = torch.empty((1, 64, 8, 8), dtype=torch.int32, device=dev)
    with pytest.raises(M.MinwError):
        M.minw_conv_block_codes_ex(act, 1, 64, 8, 8, 1, wgt, 64, 3, 3, 1, 1, 1, 0, None, None,
                                   in_format=M.CODES_E2M1, acc_out=acc)


@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 2), (3, 3)])
def test_convnet_e2m1_layers(dev, M, bits_a, bits_w):
    """A network whose hidden layers have 128-channel multiples runs them on
    E2M1 operands (the first layer writes E2M1 codes); its logits equal the
    oracle's and the E4M3-only plan's bit for bit."""
    net_p = convnet_params(53, bits_a=bits_a, bits_w=bits_w, widths=(128, 128, 256, 256),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(54, 7, hw=16)
    outs = []
    for variant in (M.VARIANT_TC_E2M1, M.VARIANT_TC_E4M3):
        net = M.Net(M.layer_descs(net_p, dev), max_batch=7, variant=variant)
        logits = torch.empty((7, net.out_features), dtype=torch.float32, device=dev)
        net.forward(dev_tensor(x, dev), logits)
        torch.cuda.synchronize()
        outs.append((logits.cpu().numpy(), net.layer_variants()))
        net.close()
    (got, var4), (got8, var8) = outs
    assert list(var4[1:]) == [M.VARIANT_TC_E2M1] * (len(var4) - 1)
    assert list(var8[1:]) == [M.VARIANT_TC] * (len(var8) - 1)
    ref = N.convnet_forward(net_p, x)
    assert np.array_equal(got, ref)
    assert np.array_equal(got8, ref)
    assert M.minw_get_last_device_error() == M.MINW_OK


def test_convnet_measured_formats(dev, M):
    """VARIANT_AUTO times every layer with E4M3 operands, E2M1 operands, E2M1
    CTA pairs, E2M1 single-CTA 128-channel tiles and the popcount path at
    creation and keeps the fastest: whatever it picks, each layer reports one
    of them, and the logits equal the oracle's bit for bit."""
    net_p = convnet_params(55, bits_a=1, bits_w=1, widths=(128, 128, 256, 256),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(56, 9, hw=16)
    net = M.Net(M.layer_descs(net_p, dev), max_batch=9, variant=M.VARIANT_AUTO)
    logits = torch.empty((9, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    var = net.layer_variants()
    net.close()
    assert all(v in (M.VARIANT_TC, M.VARIANT_TC_E2M1, M.VARIANT_TC_E2M1_PAIRS, M.VARIANT_TC_E2M1_N128,
                     M.VARIANT_POPC) for v in var[1:])
    assert np.array_equal(logits.cpu().numpy(), N.convnet_forward(net_p, x))
    assert M.minw_get_last_device_error() == M.MINW_OK


@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 1), (3, 3)])
@pytest.mark.parametrize("batch", [5, 24])
def test_convnet_e2m1_pairs(dev, M, bits_a, bits_w, batch):
    """E2M1 layers as CTA pairs of 256 pixels x 128 channels (two accumulators
    per CTA), pooled and unpooled, fully connected included, on a batch whose
    pixel tiles leave an odd pair: the logits equal the oracle's bit for bit,
    and every layer that allows it reports the pair plan."""
    net_p = convnet_params(57, bits_a=bits_a, bits_w=bits_w, widths=(128, 256, 256, 256),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(58, batch, hw=16)
    net = M.Net(M.layer_descs(net_p, dev), max_batch=batch, variant=M.VARIANT_TC_E2M1_PAIRS)
    logits = torch.empty((batch, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    var = net.layer_variants()
    net.close()
    assert M.minw_get_last_device_error() == M.MINW_OK
    assert M.VARIANT_TC_E2M1_PAIRS in list(var[1:])
    assert np.array_equal(logits.cpu().numpy(), N.convnet_forward(net_p, x))


@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 2), (3, 3)])
@pytest.mark.parametrize("batch", [7, 32])
def test_convnet_e2m1_n128(dev, M, bits_a, bits_w, batch):
    """E2M1 layers on single CTAs with 128-channel tiles (two accumulators per
    CTA at half the MMA width) for every layer with more than 128 output
    channels, pooled and unpooled, the fully connected layer included: the
    logits equal the oracle's bit for bit, and those layers report the plan."""
    net_p = convnet_params(59, bits_a=bits_a, bits_w=bits_w, widths=(128, 256, 256, 384),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(60, batch, hw=16)
    net = M.Net(M.layer_descs(net_p, dev), max_batch=batch, variant=M.VARIANT_TC_E2M1_N128)
    logits = torch.empty((batch, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    var = net.layer_variants()
    net.close()
    assert M.minw_get_last_device_error() == M.MINW_OK
    assert var[1:].count(M.VARIANT_TC_E2M1_N128) >= 3, var
    assert np.array_equal(logits.cpu().numpy(), N.convnet_forward(net_p, x))
