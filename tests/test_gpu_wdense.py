"""GPU parity of the weight-only DenseNet-BC of Table III (DenseNet-100 for
16 layers per block, growth 12, 3-bit weights), minw_wdense_create +
minw_forward, against the oracle, layer by layer on the GPU's own features
(each block's feature buffer, read back after the forward through
minw_wdense_features: block b's final features hold every layer's input and
output).

- The stem (fp32 fmaf chain, BN, HardTanh, bf16) equals the oracle's bit for
  bit.
- Each layer is recomputed by the oracle from the GPU's features before it
  (the first c channels of its block's buffer).  Its new channels may differ
  from the oracle's by at most: the fp32-accumulation bound of the 1x1
  convolution over its zero-padded channels, carried through HardTanh
  (1-Lipschitz) and the bf16 rounding of the 3x3's input (one bf16 ulp,
  2^-7 |h|, where the two roundings land on different sides), then through
  the 3x3 convolution and its own bound, HardTanh, and the bf16 rounding of
  the stored features (one more ulp).  Nearly all of them are equal bit for
  bit (the test asks for 90 %).
- Each transition likewise: its convolution's bound through HardTanh, the
  2x2 average (the same fp32 order on both sides: the bound averaged, plus
  the roundings of three fp32 adds per side, 6 x 2^-24 of the sum of
  magnitudes), and the bf16 rounding.
- The head (average pool of the bf16 features, fp32 fmaf chain, BN) on the
  GPU's last features equals the oracle's bit for bit."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import wdense_params, wresnet_input  # noqa: E402
from tests._bounds import conv_bound  # noqa: E402
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


def _pad64(c):
    return (c + 63) // 64 * 64


def _finals(net_p):
    """Each block's final channel count."""
    k = net_p["growth"]
    return [lay[-1]["b"]["w"].shape[1] + k for lay in net_p["blocks"]]


def _run(dev, M, net_p, x):
    B, hw = x.shape[0], net_p["hw"]
    net = M.Net.wdense(net_p, B, dev)
    logits = torch.empty((B, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    feats = []
    for b, cf in enumerate(_finals(net_p)):
        h = hw >> b
        t = torch.empty(B * h * h * _pad64(cf), dtype=torch.int16, device=dev)
        c, row = net.wdense_features(b, t)
        assert (c, row) == (cf, _pad64(cf))
        u = t.cpu().numpy().view(np.uint16).astype(np.uint32) << 16
        f = u.view(np.float32).reshape(B, h, h, row)[..., :c]
        feats.append(np.ascontiguousarray(f.transpose(0, 3, 1, 2)))
    out = logits.cpu().numpy()
    net.close()
    assert M.minw_get_last_device_error() == M.MINW_OK
    return out, feats


def _check_layer(lay, Fin, new_gpu, bits, thr):
    """One layer's k new channels from the GPU against the oracle recomputed
    from the GPU's features Fin before the layer (bf16 values)."""
    xb = Fin.astype(np.float64)
    y1 = N.wconv(lay["b"], Fin, 1, bits, thr)
    e1 = conv_bound(lay["b"], xb, y1, 1, bits, thr, channels=_pad64(Fin.shape[1]))
    h = O.hardtanh(y1)
    hb = O.bf16_round(h).astype(np.float64)
    dx = e1 + 2.0 ** -7 * (np.abs(h) + e1)                 # HardTanh, then one bf16 ulp
    y2 = N.wconv(lay["c"], h, 1, bits, thr)
    e2 = conv_bound(lay["c"], hb, y2, 1, bits, thr, dx=dx, channels=_pad64(h.shape[1]))
    n = O.hardtanh(y2).astype(np.float64)
    ref = O.bf16_round(O.hardtanh(y2)).astype(np.float64)
    assert np.array_equal(ref, N.wdense_layer(lay, Fin, bits, thr)[1])
    bound = e2 + 2.0 ** -7 * (np.abs(n) + e2) + 1e-30
    err = np.abs(new_gpu.astype(np.float64) - ref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound):.3f}"
    return np.mean(err == 0)


def _check_trans(tr, Fb, nxt_gpu, bits, thr):
    y = N.wconv(tr, Fb, 1, bits, thr)
    e = conv_bound(tr, Fb.astype(np.float64), y, 1, bits, thr, channels=_pad64(Fb.shape[1]))
    t = np.abs(O.hardtanh(y).astype(np.float64))
    quad = lambda a: a[:, :, 0::2, 0::2] + a[:, :, 0::2, 1::2] + a[:, :, 1::2, 0::2] + a[:, :, 1::2, 1::2]
    es, S = quad(e), quad(t)
    pe = 0.25 * (es + 6 * 2.0 ** -24 * (S + es))
    ref = N.wdense_transition(tr, Fb, bits, thr).astype(np.float64)
    bound = pe + 2.0 ** -7 * (np.abs(ref) + pe) + 1e-30
    err = np.abs(nxt_gpu.astype(np.float64) - ref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound):.3f}"
    return np.mean(err == 0)


def _check_net(net_p, x, logits, feats, pick):
    """Stem, layers and transitions of images `pick`; the head of all."""
    bits, thr, k = net_p["bits_w"], net_p["thr_w"], net_p["growth"]
    st = net_p["stem"]
    stem = O.bf16_round(O.hardtanh(O.affine(O.conv2d_f32_seq(x[pick], st["w"], 1, 1), st["scale"], st["shift"])))
    c0 = 2 * k
    assert np.array_equal(feats[0][pick, :c0], stem)
    same = []
    for b, lay_list in enumerate(net_p["blocks"]):
        Fb = feats[b][pick]
        for lay in lay_list:
            c = lay["b"]["w"].shape[1]
            same.append(_check_layer(lay, Fb[:, :c], Fb[:, c:c + k], bits, thr))
        if b < 2:
            nxt = feats[b + 1][pick]
            same.append(_check_trans(net_p["trans"][b], Fb, nxt[:, :Fb.shape[1] // 2], bits, thr))
    assert min(same) >= 0.9, f"bit-equal fractions {min(same):.3f} .. {max(same):.3f}"
    assert np.array_equal(logits, N.wresnet_head(net_p, feats[2]))       # every image's head


@pytest.mark.parametrize("layers,growth,bits,hw,B", [(3, 12, 3, 16, 3), (2, 8, 2, 8, 2), (2, 16, 1, 16, 2)])
def test_wdense_small(dev, M, layers, growth, bits, hw, B):
    """Small DenseNet-BCs (growth 12 as DenseNet-100; growth 8; growth 16,
    whose blocks end on exactly 64 channels, rows without padding): every
    layer, transition and the head against the oracle."""
    net_p = wdense_params(81 + layers + growth + bits, layers=layers, growth=growth, bits_w=bits, classes=10, hw=hw)
    x = wresnet_input(82 + growth, B, hw=hw)
    logits, feats = _run(dev, M, net_p, x)
    _check_net(net_p, x, logits, feats, list(range(B)))


def test_wdense100_sampled(dev, M):
    """DenseNet-100 (16 layers per block, growth 12, 3-bit weights) at batch
    16: all 16 images through the GPU, images 0 and 15 layer by layer
    against the oracle (each layer recomputed from the GPU's features before
    it), and the head of every image."""
    B = 16
    net_p = wdense_params(100, layers=16, growth=12, bits_w=3, classes=10, hw=32)
    x = wresnet_input(101, B, hw=32)
    logits, feats = _run(dev, M, net_p, x)
    pick = [0, B - 1]
    _check_net(net_p, x, logits, feats, pick)


def test_wdense_replay_and_batch(dev, M):
    """The same logits bit for bit on a graph replay and for a smaller batch
    than the net was created for (images 0 .. 2 of 5); the feature query
    refuses a net without a forward."""
    net_p = wdense_params(83, layers=2, growth=12, bits_w=3, classes=10, hw=16)
    x = wresnet_input(84, 5, hw=16)
    net = M.Net.wdense(net_p, 5, dev)
    with pytest.raises(M.MinwError):
        net.wdense_features(0, torch.empty(5 * 16 * 16 * 64, dtype=torch.int16, device=dev))
    outs = []
    for B in (5, 5, 3):
        logits = torch.empty((B, 10), dtype=torch.float32, device=dev)
        net.forward(dev_tensor(x[:B], dev), logits)
        torch.cuda.synchronize()
        outs.append(logits.cpu().numpy())
    net.close()
    assert np.array_equal(outs[0], outs[1]) and np.array_equal(outs[2], outs[0][:3])
