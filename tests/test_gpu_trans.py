"""GPU parity of the channel-major tensor-core tiles (128 output channels x
256 pixels, used for 64- and 128-channel layers whose only output is the next
layer's levels; a 64-channel layer loads its weight rows twice, or pads with
zero rows with the plan option dup_weights = 0): 128 -> 128 and 64 -> 64 convolutions with and
without the 2x2 pool, for each output bit width, residual blocks, against the
oracle's levels, planes and codes."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem  # noqa: E402
from tests._gpu import dev_tensor, planes_view  # noqa: E402

pytestmark = pytest.mark.gpu

# codes of the levels in integer units
_CODE = {0: 0x00, 1: 0x38, 2: 0x40, 4: 0x48, -1: 0xB8, -2: 0xC0, -4: 0xC8}


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


@pytest.mark.parametrize("ch", [128, 64])
@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("pool", [0, 1])
def test_channel_major_tiles(dev, M, bits, pool, ch):
    # 160 images of 32x32: 640 pixel tiles of 256 (>= 4 per SM), blocks that tile the image exactly;
    # the images are independent, so the oracle checks three of them
    B, C, H, W, O_ = 160, ch, 32, 32, ch
    p = conv_problem(300 + bits + 10 * pool + ch, B, C, H, W, O_, bits_a=bits, bits_w=bits, x_dist="normal",
                     w_sigma=0.05)
    a8 = torch.empty((B, H, W, C), dtype=torch.uint8, device=dev)
    w8 = torch.empty((O_, 3, 3, C), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(bits, p["thr_a"]), a8)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(bits, p["thr_w"]), w8,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    Hp, Wp = (H // 2, W // 2) if pool else (H, W)
    codes = torch.empty((B, Hp, Wp, O_), dtype=torch.uint8, device=dev)
    planes = torch.empty(M.packed_words(B, O_, Hp, Wp, bits), dtype=torch.int32, device=dev)
    qo = M.quant(bits, DEFAULT_THR[bits])
    for out in ("codes", "planes"):
        M.minw_conv_block_codes(a8, B, C, H, W, bits, w8, O_, 3, 3, bits, 1, 1, pool, dev_tensor(p["scale"], dev),
                                dev_tensor(p["shift"], dev), q_out=qo,
                                codes_out=codes if out == "codes" else None,
                                planes_out=planes if out == "planes" else None)
    torch.cuda.synchronize()
    assert M.minw_get_last_device_error() == M.MINW_OK
    pick = [0, 77, B - 1]
    al = O.quantize(p["x"][pick], bits, p["thr_a"])
    wl = O.quantize(p["w"], bits, p["thr_w"], p["w_scale"])
    acc = O.conv2d_levels(al, wl, 1, 1, bits, bits)
    if pool:
        acc = O.maxpool_i32(acc, 2, 2)
    y = O.hardtanh(O.affine(acc, p["scale"], p["shift"]))
    lv = O.quantize(y, bits, DEFAULT_THR[bits])
    units = np.rint(lv * (4 if bits == 3 else 1)).astype(int)
    want_codes = np.vectorize(_CODE.get)(units.transpose(0, 2, 3, 1)).astype(np.uint8)
    assert np.array_equal(codes.cpu().numpy()[pick], want_codes)
    assert np.array_equal(planes_view(planes, B, Hp, Wp, bits, O_)[pick], O.pack(lv, bits))


@pytest.mark.parametrize("ch", [128, 64])
@pytest.mark.parametrize("bits", [1, 2, 3])
@pytest.mark.parametrize("shortcut", ["codes", "f32"])
def test_channel_major_residual(dev, M, bits, ch, shortcut):
    """Residual block in channel-major tiles: y = fmaf(acc, scale, shift) +
    shortcut, HardTanh, quantize; the shortcut is a level-code tensor (identity
    path) or fp32 NHWC (downsample path).  Each lane holds one channel, so the
    shortcut of pixel j comes through lane j's pixel index.  A 64-channel layer
    loads its weight rows twice, so that each epilogue warp takes 64 pixel
    columns of 32 channels."""
    B, C, H, W, O_ = 160, ch, 32, 32, ch
    p = conv_problem(500 + bits + ch, B, C, H, W, O_, bits_a=bits, bits_w=bits, x_dist="normal", w_sigma=0.05)
    a8 = torch.empty((B, H, W, C), dtype=torch.uint8, device=dev)
    w8 = torch.empty((O_, 3, 3, C), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(bits, p["thr_a"]), a8)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(bits, p["thr_w"]), w8,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    qo = M.quant(bits, DEFAULT_THR[bits])
    r = np.random.default_rng(600 + bits + ch)
    if shortcut == "codes":
        xs = (r.standard_normal((B, O_, H, W)) * 0.7).astype(np.float32)
        res = O.quantize(xs, bits, DEFAULT_THR[bits]).astype(np.float32)
        res_codes = torch.empty((B, H, W, O_), dtype=torch.uint8, device=dev)
        M.aqe_quantize_codes(dev_tensor(xs, dev), qo, res_codes)
        kw = dict(res_codes=res_codes, res_bits=bits)
    else:
        res = (r.standard_normal((B, O_, H, W)) * 0.5).astype(np.float32)
        kw = dict(res_f32=dev_tensor(res.transpose(0, 2, 3, 1), dev))
    codes = torch.empty((B, H, W, O_), dtype=torch.uint8, device=dev)
    planes = torch.empty(M.packed_words(B, O_, H, W, bits), dtype=torch.int32, device=dev)
    for out in ("codes", "planes"):
        M.minw_conv_block_codes_ex(a8, B, C, H, W, bits, w8, O_, 3, 3, bits, 1, 1, 0, dev_tensor(p["scale"], dev),
                                   dev_tensor(p["shift"], dev), q_out=qo,
                                   codes_out=codes if out == "codes" else None,
                                   planes_out=planes if out == "planes" else None, **kw)
    torch.cuda.synchronize()
    assert M.minw_get_last_device_error() == M.MINW_OK
    pick = [0, 77, B - 1]
    al = O.quantize(p["x"][pick], bits, p["thr_a"])
    wl = O.quantize(p["w"], bits, p["thr_w"], p["w_scale"])
    acc = O.conv2d_levels(al, wl, 1, 1, bits, bits)
    y = O.hardtanh((O.affine(acc, p["scale"], p["shift"]) + res[pick]).astype(np.float32))
    lv = O.quantize(y, bits, DEFAULT_THR[bits])
    units = np.rint(lv * (4 if bits == 3 else 1)).astype(int)
    want_codes = np.vectorize(_CODE.get)(units.transpose(0, 2, 3, 1)).astype(np.uint8)
    assert np.array_equal(codes.cpu().numpy()[pick], want_codes)
    assert np.array_equal(planes_view(planes, B, H, W, bits, O_)[pick], O.pack(lv, bits))


def test_channel_major_zero_rows(dev, M):
    """Plan option dup_weights = 0: 64-channel tiles padded with zero weight
    rows give the same levels."""
    M.set_plan_options(dup_weights=0)
    try:
        for bits in (1, 3):
            test_channel_major_tiles(dev, M, bits, 1, 64)
    finally:
        M.set_plan_options()
