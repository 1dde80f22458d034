"""GPU parity of the CTA-pair tensor-core tiles (cta_group::2: one MMA of
256 pixels x 256 channels per pair of SMs, each CTA holding its 128 pixels and
half of the weight rows), used for 256-channel layers with K loops of at
least 18 K blocks: accumulators for several bit widths and strides with an
odd number of pixel tiles (the pair's second tile is padding), the fused
pooled block epilogue, and the same shapes with the pairs turned off."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem  # noqa: E402
from tests._gpu import dev_tensor, planes_view  # noqa: E402

pytestmark = pytest.mark.gpu

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


def _operands(dev, M, p):
    act = torch.empty((p["B"], p["H"], p["W"], p["C"]), dtype=torch.uint8, device=dev)
    wgt = torch.empty((p["O"], p["kh"], p["kw"], p["C"]), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(p["bits_a"], p["thr_a"]), act)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(p["bits_w"], p["thr_w"]), wgt,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    return act, wgt


def _ref_acc(p):
    al = O.quantize(p["x"], p["bits_a"], p["thr_a"])
    wl = O.quantize(p["w"], p["bits_w"], p["thr_w"], p["w_scale"])
    return O.conv2d_levels(al, wl, p["stride"], p["pad"], p["bits_a"], p["bits_w"])


# (B, C, H, W, O, stride): 3, 1, 1 and 1 pixel tiles (odd: one padding tile per channel tile)
CASES = [(3, 256, 10, 10, 512, 1), (2, 512, 7, 7, 256, 1), (2, 256, 14, 14, 512, 2)]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("ba,bw", [(1, 1), (2, 1), (3, 3)])
def test_pair_accumulators(dev, M, case, ba, bw):
    B, C, H, W, O_, s = case
    p = conv_problem(700 + 10 * ba + bw + C // 64, B, C, H, W, O_, 3, 3, s, 1, ba, bw, w_sigma=0.5)
    act, wgt = _operands(dev, M, p)
    Ho, Wo = (H + 2 - 3) // s + 1, (W + 2 - 3) // s + 1
    acc = torch.full((B, O_, Ho, Wo), -7, dtype=torch.int32, device=dev)
    M.minw_conv2d_codes(act, B, C, H, W, ba, wgt, O_, 3, 3, bw, s, 1, acc_out=acc)
    torch.cuda.synchronize()
    assert M.minw_get_last_device_error() == M.MINW_OK
    ref = _ref_acc(p)
    got = acc.cpu().numpy()
    assert np.array_equal(got, ref), f"{np.sum(got != ref)} of {ref.size} accumulators differ"


@pytest.mark.parametrize("bits", [1, 3])
def test_pair_pooled_block(dev, M, bits):
    # 256 -> 256, 16 x 16, 2x2 pool: the level-mask epilogue on each CTA's own 128 pixels
    B, C, H, W, O_ = 12, 256, 16, 16, 256
    p = conv_problem(800 + bits, B, C, H, W, O_, bits_a=bits, bits_w=bits, x_dist="normal", w_sigma=0.05)
    act, wgt = _operands(dev, M, p)
    qo = M.quant(bits, DEFAULT_THR[bits])
    codes = torch.empty((B, H // 2, W // 2, O_), dtype=torch.uint8, device=dev)
    planes = torch.empty(M.packed_words(B, O_, H // 2, W // 2, bits), dtype=torch.int32, device=dev)
    for out in ("codes", "planes"):
        M.minw_conv_block_codes(act, B, C, H, W, bits, wgt, O_, 3, 3, bits, 1, 1, 1, dev_tensor(p["scale"], dev),
                                dev_tensor(p["shift"], dev), q_out=qo,
                                codes_out=codes if out == "codes" else None,
                                planes_out=planes if out == "planes" else None)
    torch.cuda.synchronize()
    assert M.minw_get_last_device_error() == M.MINW_OK
    acc = O.maxpool_i32(_ref_acc(p), 2, 2)
    y = O.hardtanh(O.affine(acc, p["scale"], p["shift"]))
    lv = O.quantize(y, bits, DEFAULT_THR[bits])
    units = np.rint(lv * (4 if bits == 3 else 1)).astype(int)
    want = np.vectorize(_CODE.get)(units.transpose(0, 2, 3, 1)).astype(np.uint8)
    assert np.array_equal(codes.cpu().numpy(), want)
    assert np.array_equal(planes_view(planes, B, H // 2, W // 2, bits, O_), O.pack(lv, bits))


def test_pairs_off(dev):
    """Plan option cta_pairs = 0: the same shapes on single-CTA tiles give the
    same accumulators."""
    from paper_2003_04296_gb300 import minw
    minw.set_plan_options(cta_pairs=0)
    try:
        for (B, C, H, W, O_, s) in CASES:
            p = conv_problem(900 + C // 64, B, C, H, W, O_, 3, 3, s, 1, 2, 2, w_sigma=0.5)
            act, wgt = _operands(dev, minw, p)
            Ho, Wo = (H - 1) // s + 1, (W - 1) // s + 1
            acc = torch.empty((B, O_, Ho, Wo), dtype=torch.int32, device=dev)
            minw.minw_conv2d_codes(act, B, C, H, W, 2, wgt, O_, 3, 3, 2, s, 1, acc_out=acc)
            torch.cuda.synchronize()
            assert minw.minw_get_last_device_error() == minw.MINW_OK
            assert np.array_equal(acc.cpu().numpy(), _ref_acc(p))
    finally:
        minw.set_plan_options()
