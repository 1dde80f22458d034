"""GPU parity at the full sizes of the workloads, through the C ABI:
- a single 3x3 convolution, 4x128x32x32, 1-bit x 1-bit, int32 accumulators and
  the fp32 scale epilogue, every output checked (popcount and tensor-core paths);
- the bit-width sweep 256x512x14x14 -> 512 channels, (M, N) in {1,2,3}^2, on the
  tensor-core path, with images 0 and 255 re-computed by the oracle (the
  images of a batch are independent);
- AQE forward/backward and quantize + pack on the full 256x512x14x14 tensor;
- the CIFAR ConvNet with 2-bit activations x 1- and 2-bit weights at batch 256,
  images 0 and 255 re-run by the oracle, and one layer fed |N(0,1)| clipped
  to [0, 1] activations."""
from itertools import product

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import (DEFAULT_THR, aqe_problem, conv_problem, convnet_input,  # noqa: E402
                                           convnet_params)
from tests._gpu import assert_close, dev_tensor, planes_view  # noqa: E402

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


def _levels(p):
    al = O.quantize(p["x"], p["bits_a"], p["thr_a"])
    wl = O.quantize(p["w"], p["bits_w"], p["thr_w"], p["w_scale"])
    return al, wl


def test_single_conv_4x128x32x32_both_paths(dev, M):
    p = conv_problem(0, 4, 128, 32, 32, 128, 3, 3, 1, 1, 1, 1, w_sigma=0.05)
    al, wl = _levels(p)
    ref = O.conv2d_levels(al, wl, 1, 1, 1, 1)
    yref = O.affine(ref, p["scale"], p["shift"])
    x, w = dev_tensor(p["x"], dev), dev_tensor(p["w"], dev)
    sc, sh = dev_tensor(p["scale"], dev), dev_tensor(p["shift"], dev)
    # popcount path on bit-planes
    act = torch.empty(M.packed_words(4, 128, 32, 32, 1), dtype=torch.int32, device=dev)
    wgt = torch.empty(M.packed_words(128, 128, 3, 3, 1), dtype=torch.int32, device=dev)
    M.aqe_quantize_pack(x, M.quant(1), act)
    M.minw_pack_weights(w, M.quant(1), wgt, channel_scale=dev_tensor(p["w_scale"], dev))
    acc = torch.empty((4, 128, 32, 32), dtype=torch.int32, device=dev)
    y = torch.empty((4, 128, 32, 32), dtype=torch.float32, device=dev)
    M.minw_conv2d(act, 4, 128, 32, 32, 1, wgt, 128, 3, 3, 1, 1, 1, acc_out=acc, scale=sc, shift=sh, y_out=y,
                  variant=M.VARIANT_POPC)
    assert np.array_equal(acc.cpu().numpy(), ref)
    assert np.array_equal(y.cpu().numpy(), yref)
    # tensor-core path on level codes
    a8 = torch.empty((4, 32, 32, 128), dtype=torch.uint8, device=dev)
    w8 = torch.empty((128, 3, 3, 128), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(x, M.quant(1), a8)
    M.minw_pack_weight_codes(w, M.quant(1), w8, channel_scale=dev_tensor(p["w_scale"], dev))
    acc.fill_(-7)
    M.minw_conv2d_codes(a8, 4, 128, 32, 32, 1, w8, 128, 3, 3, 1, 1, 1, acc_out=acc, scale=sc, shift=sh, y_out=y)
    assert np.array_equal(acc.cpu().numpy(), ref)
    assert np.array_equal(y.cpu().numpy(), yref)


@pytest.fixture(scope="module")
def sweep_input():
    return conv_problem(5, 256, 512, 14, 14, 512, 3, 3, 1, 1, 1, 1, x_dist="normal", w_sigma=1.0)


@pytest.mark.parametrize("ba,bw", list(product([1, 2, 3], [1, 2, 3])))
def test_bitwidth_sweep_256x512x14x14(dev, M, sweep_input, ba, bw):
    base = sweep_input
    p = dict(base, bits_a=ba, bits_w=bw, thr_a=DEFAULT_THR[ba], thr_w=DEFAULT_THR[bw],
             w_scale=(np.ones(512, np.float32) if bw == 1 else
                      (1.0 / np.abs(base["w"].reshape(512, -1)).max(1)).astype(np.float32)))
    x, w = dev_tensor(p["x"], dev), dev_tensor(p["w"], dev)
    a8 = torch.empty((256, 14, 14, 512), dtype=torch.uint8, device=dev)
    w8 = torch.empty((512, 3, 3, 512), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(x, M.quant(ba, p["thr_a"]), a8)
    M.minw_pack_weight_codes(w, M.quant(bw, p["thr_w"]), w8, channel_scale=dev_tensor(p["w_scale"], dev))
    acc = torch.empty((256, 512, 14, 14), dtype=torch.int32, device=dev)
    M.minw_conv2d_codes(a8, 256, 512, 14, 14, ba, w8, 512, 3, 3, bw, 1, 1, acc_out=acc)
    got = acc.cpu().numpy()
    wl = O.quantize(p["w"], bw, p["thr_w"], p["w_scale"])
    for i in (0, 255):
        al = O.quantize(p["x"][i:i + 1], ba, p["thr_a"])
        ref = O.conv2d_levels(al, wl, 1, 1, ba, bw)
        assert np.array_equal(got[i:i + 1], ref), f"image {i}: {np.sum(got[i:i + 1] != ref)} accumulators differ"
    assert M.minw_get_last_device_error() == M.MINW_OK


def test_aqe_and_pack_full_tensor(dev, M):
    """AQE fwd/bwd (alpha = 0.75) and the fused quantize + pack on the
    256x512x14x14 activation tensor (25.7 M elements)."""
    n = 256 * 512 * 14 * 14
    p = aqe_problem(5, n, alpha=0.75)
    x = dev_tensor(p["x"], dev)
    g = dev_tensor(p["g"], dev)
    y = torch.empty_like(x)
    gx = torch.empty_like(x)
    for bits in (1, 2, 3):
        M.aqe_forward(x, y, 0.75, M.quant(bits, DEFAULT_THR[bits]))
        assert_close(y.cpu().numpy(), O.aqe_forward(p["x"], 0.75, bits, DEFAULT_THR[bits]))
    M.aqe_backward(x, g, gx, 0.75)
    assert_close(gx.cpu().numpy(), O.aqe_backward(p["x"], p["g"], 0.75))
    x4 = x.view(256, 512, 14, 14)
    planes = torch.empty(M.packed_words(256, 512, 14, 14, 3), dtype=torch.int32, device=dev)
    M.aqe_quantize_pack(x4, M.quant(3, DEFAULT_THR[3]), planes)
    lv = O.quantize(p["x"].reshape(256, 512, 14, 14)[:8], 3, DEFAULT_THR[3])
    assert np.array_equal(planes_view(planes, 256, 14, 14, 3, 512)[:8], O.pack(lv, 3))


@pytest.mark.parametrize("bits_w", [1, 2])
def test_cifar_convnet_2bit_activations_batch256(dev, M, bits_w):
    net_p = convnet_params(3, bits_a=2, bits_w=bits_w)
    x = convnet_input(3, 256)
    net = M.Net(M.layer_descs(net_p, dev), max_batch=256)
    logits = torch.empty((256, 10), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    got = logits.cpu().numpy()
    net.close()
    for i in (0, 255):
        assert np.array_equal(got[i:i + 1], N.convnet_forward(net_p, x[i:i + 1]))


def test_clipped_abs_normal_activations_layer(dev, M):
    """One 2-bit x 2-bit layer at the ConvNet's second-layer shape fed
    |N(0,1)| clipped to [0, 1] (every sign bit 0), batch 256, block epilogue
    with pooling; images 0 and 255 checked."""
    p = conv_problem(33, 256, 128, 32, 32, 128, 3, 3, 1, 1, 2, 2, x_dist="absnormal_clip", w_sigma=0.05)
    x, w = dev_tensor(p["x"], dev), dev_tensor(p["w"], dev)
    a8 = torch.empty((256, 32, 32, 128), dtype=torch.uint8, device=dev)
    w8 = torch.empty((128, 3, 3, 128), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(x, M.quant(2, DEFAULT_THR[2]), a8)
    M.minw_pack_weight_codes(w, M.quant(2, DEFAULT_THR[2]), w8, channel_scale=dev_tensor(p["w_scale"], dev))
    y = torch.empty((256, 128, 16, 16), dtype=torch.float32, device=dev)
    codes = torch.empty((256, 16, 16, 128), dtype=torch.uint8, device=dev)
    M.minw_conv_block_codes(a8, 256, 128, 32, 32, 2, w8, 128, 3, 3, 2, 1, 1, 1, dev_tensor(p["scale"], dev),
                            dev_tensor(p["shift"], dev), q_out=M.quant(2, DEFAULT_THR[2]), codes_out=codes,
                            y_out=y)
    got = y.cpu().numpy()
    wl = O.quantize(p["w"], 2, DEFAULT_THR[2], p["w_scale"])
    for i in (0, 255):
        al = O.quantize(p["x"][i:i + 1], 2, DEFAULT_THR[2])
        assert np.all(al >= 0)
        acc = O.maxpool_i32(O.conv2d_levels(al, wl, 1, 1, 2, 2), 2, 2)
        yr = O.hardtanh(O.affine(acc, p["scale"], p["shift"]))
        assert np.array_equal(got[i:i + 1], yr)
