"""GPU parity of the tensor-core path (level codes + tcgen05 FP8 contraction)
against the oracle, through the C ABI: the codes layout, the convolution for
all nine bit-width pairs on ragged tiles, the fused block epilogue, and
accumulators at the largest magnitudes the workloads reach."""
from itertools import product

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem  # noqa: E402
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


def decode_e4m3(b):
    """FP8 E4M3 bytes to values from the format's definition (1 sign bit,
    4 exponent bits with bias 7, 3 mantissa bits); normal numbers only plus 0."""
    b = b.astype(np.int64)
    sign = np.where(b & 0x80, -1.0, 1.0)
    e = (b >> 3) & 0xF
    m = b & 7
    v = sign * (1.0 + m / 8.0) * np.power(2.0, e - 7.0)
    return np.where((b & 0x7F) == 0, 0.0, v)


@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("shape", [(2, 128, 5, 7), (1, 48, 3, 3), (3, 16, 1, 1)])
def test_quantize_codes(dev, M, bits, shape):
    B, C, H, W = shape
    x = np.random.default_rng(C + bits).standard_normal(shape).astype(np.float32)
    codes = torch.empty((B, H, W, C), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(x, dev), M.quant(bits, DEFAULT_THR[bits]), codes)
    lv = O.quantize(x, bits, DEFAULT_THR[bits]) * 2.0 ** O.units_shift(bits)
    assert np.array_equal(decode_e4m3(codes.cpu().numpy()), lv.transpose(0, 2, 3, 1))


@pytest.mark.parametrize("bits", [1, 2, 3])
def test_weight_codes(dev, M, bits):
    w = np.random.default_rng(bits).normal(0, 0.05, (40, 256, 3, 3)).astype(np.float32)
    cs = (1.0 / np.abs(w.reshape(40, -1)).max(1)).astype(np.float32)
    codes = torch.empty((40, 3, 3, 256), dtype=torch.uint8, device=dev)
    M.minw_pack_weight_codes(dev_tensor(w, dev), M.quant(bits, DEFAULT_THR[bits]), codes,
                             channel_scale=dev_tensor(cs, dev))
    lv = O.quantize(w, bits, DEFAULT_THR[bits], cs) * 2.0 ** O.units_shift(bits)
    assert np.array_equal(decode_e4m3(codes.cpu().numpy()), lv.transpose(0, 2, 3, 1))


def _operands(dev, M, p):
    B, C, H, W, O_ = p["B"], p["C"], p["H"], p["W"], p["O"]
    act = torch.empty((B, H, W, C), dtype=torch.uint8, device=dev)
    wgt = torch.empty((O_, p["kh"], p["kw"], C), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(p["bits_a"], p["thr_a"]), act)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(p["bits_w"], p["thr_w"]), wgt,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    return act, wgt


def _ref_acc(p):
    al = O.quantize(p["x"], p["bits_a"], p["thr_a"])
    wl = O.quantize(p["w"], p["bits_w"], p["thr_w"], p["w_scale"])
    return O.conv2d_levels(al, wl, p["stride"], p["pad"], p["bits_a"], p["bits_w"])


TC_CASES = [
    # B, C, H, W, O, k, pad
    (2, 128, 9, 7, 70, 3, 1),       # ragged rows/columns of the pixel tile, ragged O
    (3, 256, 16, 16, 256, 3, 1),    # BN = 256
    (2, 128, 8, 8, 10, 1, 0),       # O = 10 -> one 16-wide channel tile
    (130, 512, 4, 4, 20, 4, 0),     # fully connected over a 4x4 map, 2 image tiles
    (2, 128, 1, 1, 300, 1, 0),      # two channel tiles, the second ragged
    (1, 128, 14, 14, 64, 3, 1),     # 14x14: tiles overhang both edges
]


@pytest.mark.parametrize("case", TC_CASES)
@pytest.mark.parametrize("ba,bw", list(product([1, 2, 3], [1, 2, 3])))
def test_conv2d_codes(dev, M, case, ba, bw):
    B, C, H, W, O_, k, pad = case
    p = conv_problem(case_seed(case, ba, bw, "tc"), B, C, H, W, O_, k, k, 1, pad, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    acc = torch.full((B, O_, p["H"] + 2 * pad - k + 1, p["W"] + 2 * pad - k + 1), -7, dtype=torch.int32,
                     device=dev)
    y = torch.empty(acc.shape, dtype=torch.float32, device=dev)
    M.minw_conv2d_codes(act, B, C, H, W, ba, wgt, O_, k, k, bw, 1, pad, acc_out=acc,
                        scale=dev_tensor(p["scale"], dev), shift=dev_tensor(p["shift"], dev), y_out=y)
    ref = _ref_acc(p)
    got = acc.cpu().numpy()
    assert np.array_equal(got, ref), f"{np.sum(got != ref)} of {ref.size} accumulators differ"
    assert np.array_equal(y.cpu().numpy(), O.affine(ref, p["scale"], p["shift"]))
    assert M.minw_get_last_device_error() == M.MINW_OK


@pytest.mark.parametrize("ba,bw,hw", [(1, 1, 32), (2, 2, 16), (3, 3, 8), (2, 1, 16)])
def test_conv_block_codes_pool(dev, M, ba, bw, hw):
    B, C, O_ = 2, 128, 96
    p = conv_problem(61 + ba + 3 * bw + hw, B, C, hw, hw, O_, 3, 3, 1, 1, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    bo = ba
    h2 = hw // 2
    codes = torch.full((B, h2, h2, O_), 0x77, dtype=torch.uint8, device=dev)
    planes = torch.full((M.packed_words(B, O_, h2, h2, bo),), -1, dtype=torch.int32, device=dev)
    y = torch.empty((B, O_, h2, h2), dtype=torch.float32, device=dev)
    M.minw_conv_block_codes(act, B, C, hw, hw, ba, wgt, O_, 3, 3, bw, 1, 1, 1, dev_tensor(p["scale"], dev),
                            dev_tensor(p["shift"], dev), q_out=M.quant(bo, DEFAULT_THR[bo]), codes_out=codes,
                            planes_out=planes, y_out=y)
    acc = O.maxpool_i32(_ref_acc(p), 2, 2)
    yr = O.hardtanh(O.affine(acc, p["scale"], p["shift"]))
    assert np.array_equal(y.cpu().numpy(), yr)
    lv = O.quantize(yr, bo, DEFAULT_THR[bo])
    assert np.array_equal(planes_view(planes, B, h2, h2, bo, O_), O.pack(lv, bo))
    assert np.array_equal(decode_e4m3(codes.cpu().numpy()),
                          (lv * 2.0 ** O.units_shift(bo)).transpose(0, 2, 3, 1))


def _adversarial(bits, C, k, hw, B=2, O_=64):
    """Image 0 at the largest level everywhere (all products maximal); image 1
    at the largest level on the first half of the channels and the smallest
    non-zero level on the rest, so unit products follow large partial sums.
    Even output channels use the largest weight level, odd ones mix in the
    smaller levels."""
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
def test_exact_at_largest_magnitudes(dev, M, bits, C, k, hw):
    """|acc| up to 16 * 4608 (3-bit, 512 x 3 x 3) and 8192 (1-bit FC) with
    unit products next to the largest: the fp32 tensor-core accumulator must
    reproduce every integer exactly."""
    p = _adversarial(bits, C, k, hw)
    act, wgt = _operands(dev, M, p)
    Ho = hw + 2 * p["pad"] - k + 1
    acc = torch.empty((p["B"], p["O"], Ho, Ho), dtype=torch.int32, device=dev)
    M.minw_conv2d_codes(act, p["B"], C, hw, hw, bits, wgt, p["O"], k, k, bits, 1, p["pad"], acc_out=acc)
    ref = _ref_acc(p)
    assert np.abs(ref).max() == (16 if bits == 3 else 1) * C * k * k
    assert np.array_equal(acc.cpu().numpy(), ref)


def test_codes_argument_errors(dev, M):
    """Shapes outside the tensor-core path are rejected on the host before any
    launch (the tiny buffers are never read)."""
    t = torch.empty(4096, dtype=torch.uint8, device=dev)
    a = torch.empty(64, dtype=torch.int32, device=dev)
    with pytest.raises(M.MinwError) as e1:   # C % 64 != 0
        M.minw_conv2d_codes(t, 1, 32, 4, 4, 1, t, 8, 3, 3, 1, 1, 1, acc_out=a)
    assert e1.value.status == M.MINW_EUNSUPPORTED
    with pytest.raises(M.MinwError) as e2:   # stride 3
        M.minw_conv2d_codes(t, 1, 128, 4, 4, 1, t, 8, 3, 3, 1, 3, 1, acc_out=a)
    assert e2.value.status == M.MINW_EUNSUPPORTED


def _fc_problem(seed, B, K, O, ba, bw):
    p = conv_problem(seed, B, K, 1, 1, O, 1, 1, 1, 0, ba, bw, w_sigma=0.5)
    return p


@pytest.mark.parametrize("B,K,Oc,ba,bw", [(256, 8192, 1024, 1, 1), (130, 4096, 1024, 2, 2), (256, 2048, 10, 1, 1),
                                         (64, 4096, 512, 3, 3)])
def test_fc_split_k(dev, M, B, K, Oc, ba, bw):
    """Fully connected layer with the K reduction split across CTAs: equal to
    the unsplit kernel and to the oracle, two calls in a row on one workspace
    (whose contents are garbage between calls)."""
    p = _fc_problem(B + K + Oc, B, K, Oc, ba, bw)
    act = torch.empty((B, 1, 1, K), dtype=torch.uint8, device=dev)
    wgt = torch.empty((Oc, 1, 1, K), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(ba, p["thr_a"]), act)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(bw, p["thr_w"]), wgt,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    nbytes = M.minw_fc_workspace_bytes(B, K, Oc)
    assert nbytes > 0
    ws = torch.full((nbytes,), 0x5A, dtype=torch.uint8, device=dev)
    sc, sh = dev_tensor(p["scale"], dev), dev_tensor(p["shift"], dev)
    ref = _ref_acc(p).reshape(B, Oc)
    last = Oc % 16 != 0
    q = None if last else M.quant(ba, DEFAULT_THR[ba])
    outs = []
    half = ws[: nbytes // 2]
    for use_ws in (ws, ws, half, None):
        acc = torch.full((B, Oc), -7, dtype=torch.int32, device=dev)
        y = torch.empty((B, Oc), dtype=torch.float32, device=dev)
        codes = None if last else torch.empty((B, Oc), dtype=torch.uint8, device=dev)
        M.minw_fc_codes(act, B, K, ba, wgt, Oc, bw, scale=sc, shift=sh, q_out=q, codes_out=codes, y_out=y,
                        acc_out=acc, workspace=use_ws)
        torch.cuda.synchronize()
        assert np.array_equal(acc.cpu().numpy(), ref)
        yr = O.affine(ref, p["scale"], p["shift"])
        if not last:
            yr = O.hardtanh(yr)
        assert np.array_equal(y.cpu().numpy(), yr)
        outs.append(codes.cpu().numpy() if codes is not None else None)
    if not last:
        lv = O.quantize(O.hardtanh(O.affine(ref, p["scale"], p["shift"])), ba, DEFAULT_THR[ba])
        assert np.array_equal(decode_e4m3(outs[0]), lv * 2.0 ** O.units_shift(ba))
        assert np.array_equal(outs[0], outs[2]) and np.array_equal(outs[0], outs[3])
    assert M.minw_get_last_device_error() == M.MINW_OK


TC_STRIDED = [
    # B, C, H, W, O, k, stride, pad
    (2, 64, 9, 7, 70, 3, 1, 1),       # 64-channel input: 64-byte K chunks
    (2, 128, 16, 16, 128, 3, 2, 1),   # stride 2
    (1, 128, 15, 13, 32, 3, 2, 1),    # stride 2, odd sizes
    (2, 64, 14, 14, 128, 1, 2, 0),    # 1x1 / 2 downsample, 64 channels
    (3, 64, 56, 56, 64, 3, 1, 1),     # ResNet layer-1 shape (partial tiles at the right edge)
]


@pytest.mark.parametrize("case", TC_STRIDED)
@pytest.mark.parametrize("ba,bw", [(1, 1), (3, 3), (2, 1)])
def test_conv2d_codes_strided_and_64ch(dev, M, case, ba, bw):
    B, C, H, W, O_, k, s, pad = case
    p = conv_problem(case_seed(case, ba, bw, "s"), B, C, H, W, O_, k, k, s, pad, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    Ho = (H + 2 * pad - k) // s + 1
    Wo = (W + 2 * pad - k) // s + 1
    acc = torch.full((B, O_, Ho, Wo), -7, dtype=torch.int32, device=dev)
    M.minw_conv2d_codes(act, B, C, H, W, ba, wgt, O_, k, k, bw, s, pad, acc_out=acc)
    ref = _ref_acc(p)
    got = acc.cpu().numpy()
    assert np.array_equal(got, ref), f"{np.sum(got != ref)} of {ref.size} accumulators differ"


@pytest.mark.parametrize("shortcut", ["codes", "f32"])
@pytest.mark.parametrize("bits", [3, 1])
def test_residual_block_epilogue(dev, M, shortcut, bits):
    """y = fmaf(acc, scale, shift) + shortcut (one fp32 add), HardTanh, quantize;
    the shortcut is a level-code tensor (identity path) or fp32 NHWC (the
    downsample path, itself produced by a block that writes its BN output)."""
    B, C, H, W, O_ = 2, 128, 10, 12, 128
    p = conv_problem(71 + bits, B, C, H, W, O_, 3, 3, 1, 1, bits, bits, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    sc, sh = dev_tensor(p["scale"], dev), dev_tensor(p["shift"], dev)
    acc_ref = _ref_acc(p)
    y_bn = O.affine(acc_ref, p["scale"], p["shift"])                      # NCHW fp32
    r = np.random.default_rng(5)
    if shortcut == "codes":
        xs = (r.standard_normal((B, O_, H, W)) * 0.7).astype(np.float32)
        res_lv = O.quantize(xs, bits, DEFAULT_THR[bits])                 # dequantized levels
        res_codes = torch.empty((B, H, W, O_), dtype=torch.uint8, device=dev)
        M.aqe_quantize_codes(dev_tensor(xs, dev), M.quant(bits, DEFAULT_THR[bits]), res_codes)
        kw = dict(res_codes=res_codes, res_bits=bits)
        res = res_lv.astype(np.float32)
    else:
        res = (r.standard_normal((B, O_, H, W)) * 0.5).astype(np.float32)
        kw = dict(res_f32=dev_tensor(res.transpose(0, 2, 3, 1), dev))
    y_nhwc = torch.empty((B, H, W, O_), dtype=torch.float32, device=dev)
    codes = torch.empty((B, H, W, O_), dtype=torch.uint8, device=dev)
    y = torch.empty((B, O_, H, W), dtype=torch.float32, device=dev)
    M.minw_conv_block_codes_ex(act, B, C, H, W, bits, wgt, O_, 3, 3, bits, 1, 1, 0, sc, sh,
                               q_out=M.quant(bits, DEFAULT_THR[bits]), codes_out=codes, y_out=y, y_nhwc=y_nhwc,
                               **kw)
    assert np.array_equal(y_nhwc.cpu().numpy(), y_bn.transpose(0, 2, 3, 1))
    yr = O.hardtanh((y_bn + res).astype(np.float32))
    assert np.array_equal(y.cpu().numpy(), yr)
    lv = O.quantize(yr, bits, DEFAULT_THR[bits])
    assert np.array_equal(decode_e4m3(codes.cpu().numpy()), (lv * 2.0 ** O.units_shift(bits)).transpose(0, 2, 3, 1))
