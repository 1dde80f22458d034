"""GPU parity at the full sizes of the workloads, through the C ABI:
- a single 3x3 convolution, 4x128x32x32, 1-bit x 1-bit, int32 accumulators and
  the fp32 scale epilogue, every output checked (popcount and tensor-core paths);
- the bit-width sweep 256x512x14x14 -> 512 channels, (M, N) in {1,2,3}^2, on the
  tensor-core path with E4M3 and with E2M1 operands, 16 images spread over the
  batch (so over every wave of tiles, the last partial one included)
  re-computed by the oracle (the images of a batch are independent);
- AQE forward/backward and quantize + pack on the full 256x512x14x14 tensor;
- the CIFAR ConvNet with 2-bit activations x 1- and 2-bit weights at batch 256,
  16 spread images re-run by the oracle, and one layer fed |N(0,1)| clipped
  to [0, 1] activations (16 spread images).
The oracle's runs are spread over the host's cores (tests/_oracle_pool.py)."""
from itertools import product

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import (DEFAULT_THR, aqe_problem, conv_problem, convnet_input,  # noqa: E402
                                           convnet_params)
from tests import _oracle_pool as OP  # noqa: E402
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


SWEEP_SPEC = (5, 256, 512, 14, 14, 512, 3, 1, 1, "normal", 1.0)


@pytest.fixture(scope="module")
def sweep_input():
    s = SWEEP_SPEC
    return conv_problem(s[0], s[1], s[2], s[3], s[4], s[5], s[6], s[6], s[7], s[8], 1, 1, x_dist=s[9], w_sigma=s[10])


@pytest.mark.parametrize("ba,bw", list(product([1, 2, 3], [1, 2, 3])))
def test_bitwidth_sweep_256x512x14x14(dev, M, sweep_input, ba, bw):
    base = sweep_input
    p = dict(base, bits_a=ba, bits_w=bw, thr_a=DEFAULT_THR[ba], thr_w=DEFAULT_THR[bw],
             w_scale=(np.ones(512, np.float32) if bw == 1 else
                      (1.0 / np.abs(base["w"].reshape(512, -1)).max(1)).astype(np.float32)))
    idx = OP.spread(256)
    refs = OP.starmap(OP.conv_acc, [(SWEEP_SPEC, ba, bw, "ones" if bw == 1 else "max", i) for i in idx])
    x, w = dev_tensor(p["x"], dev), dev_tensor(p["w"], dev)
    ws = dev_tensor(p["w_scale"], dev)
    acc = torch.empty((256, 512, 14, 14), dtype=torch.int32, device=dev)
    for fmt in (M.CODES_E4M3, M.CODES_E2M1):
        cb = 512 if fmt == M.CODES_E4M3 else 256
        a8 = torch.empty((256, 14, 14, cb), dtype=torch.uint8, device=dev)
        w8 = torch.empty((512, 3, 3, cb), dtype=torch.uint8, device=dev)
        if fmt == M.CODES_E4M3:
            M.aqe_quantize_codes(x, M.quant(ba, p["thr_a"]), a8)
            M.minw_pack_weight_codes(w, M.quant(bw, p["thr_w"]), w8, channel_scale=ws)
        else:
            M.aqe_quantize_codes_e2m1(x, M.quant(ba, p["thr_a"]), a8)
            M.minw_pack_weight_codes_e2m1(w, M.quant(bw, p["thr_w"]), w8, channel_scale=ws)
        acc.fill_(-7)
        M.minw_conv_block_codes_ex(a8, 256, 512, 14, 14, ba, w8, 512, 3, 3, bw, 1, 1, 0, None, None,
                                   in_format=fmt, acc_out=acc)
        got = acc.cpu().numpy()
        for i, ref in zip(idx, refs):
            assert np.array_equal(got[i:i + 1], ref), f"format {fmt}, image {i}: {np.sum(got[i:i + 1] != ref)} differ"
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
    idx = OP.spread(256)
    refs = OP.starmap(OP.convnet_logits, [(3, 2, bits_w, 3, 256, i) for i in idx])
    for i, ref in zip(idx, refs):
        assert np.array_equal(got[i:i + 1], ref), f"image {i}"


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
    assert np.all(p["x"] >= 0)
    idx = OP.spread(256)
    spec = (33, 256, 128, 32, 32, 128, 3, 1, 1, "absnormal_clip", 0.05)
    accs = OP.starmap(OP.conv_acc, [(spec, 2, 2, "max", i) for i in idx])
    for i, acc in zip(idx, accs):
        yr = O.hardtanh(O.affine(O.maxpool_i32(acc, 2, 2), p["scale"], p["shift"]))
        assert np.array_equal(got[i:i + 1], yr), f"image {i}"
