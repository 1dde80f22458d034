"""GPU parity of the weight-only residual network of Table III (a CIFAR
ResNet-(6n+2) with N-bit weights and full-precision activations; ResNet-110
for n = 18), minw_wresnet_create + minw_forward, against the oracle, stage by
stage on the GPU's own activations (kept by the net for this purpose).

- The stem (fp32 fmaf chain, BN, HardTanh) equals the oracle's bit for bit.
- Each block is recomputed by the oracle from the GPU's input to that block.
  The GPU's convolutions sum in the tensor core's order in fp32, so a block's
  output may differ from the oracle's by at most: the fp32-accumulation bound
  of conv1 (|scale| K 2^-23 sum|x w| + 2^-23 |y|), carried through HardTanh
  (1-Lipschitz) and through the bf16 rounding of conv2's input (one bf16 ulp,
  2^-7 |h|, where the two roundings land on different sides), then through
  conv2 (|scale| times the convolution of those input bounds with |w|, plus
  its own accumulation bound), the shortcut convolution's bound, and the fp32
  add.  A wrong tap, stride, channel, shortcut or HardTanh breaks it by
  orders of magnitude.
- The head (average pool, fp32 fmaf chain, BN) on the GPU's last activation
  equals the oracle's bit for bit."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import wresnet_input, wresnet_params  # noqa: E402
from tests._bounds import conv_bound as _conv_bound  # noqa: E402
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


def _check_block(blk, a, out_gpu, bits, thr):
    """Block output of the GPU against the oracle recomputed from the GPU's
    own block input a, within the bound of the module docstring."""
    ab = O.bf16_round(a).astype(np.float64)
    y1 = N.wconv(blk["c1"], a, blk["stride"], bits, thr)
    e1 = _conv_bound(blk["c1"], ab, y1, blk["stride"], bits, thr)
    h = O.hardtanh(y1)
    hb = O.bf16_round(h).astype(np.float64)
    dx = e1 + 2.0 ** -7 * (np.abs(h) + e1)               # HardTanh, then one bf16 ulp
    y2 = N.wconv(blk["c2"], h, 1, bits, thr)
    e2 = _conv_bound(blk["c2"], hb, y2, 1, bits, thr, dx=dx)
    if blk["down"] is None:
        s, es = a, 0.0
    else:
        s = N.wconv(blk["down"], a, 2, bits, thr)
        es = _conv_bound(blk["down"], ab, s, 2, bits, thr)
    ref = O.hardtanh((y2 + s).astype(np.float32))
    bound = e2 + es + 2.0 ** -22 * np.abs(y2.astype(np.float64) + s) + 1e-30
    err = np.abs(out_gpu.astype(np.float64) - ref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound):.3f}"
    return ref


def _run(dev, M, net_p, x, keep=True):
    B = x.shape[0]
    net = M.Net.wresnet(net_p, B, dev, keep_activations=keep)
    logits = torch.empty((B, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    acts = []
    if keep:
        hw = net_p["hw"]
        shapes = [(B, 16, hw, hw)]
        size = hw
        for blk in net_p["blocks"]:
            size //= blk["stride"]
            shapes.append((B, blk["c2"]["w"].shape[0], size, size))
        for i, sh in enumerate(shapes):
            t = torch.empty(sh, dtype=torch.float32, device=dev)
            net.wresnet_activation(i, t)
            acts.append(t)
        torch.cuda.synchronize()
        acts = [t.cpu().numpy() for t in acts]
    out = logits.cpu().numpy()
    net.close()
    assert M.minw_get_last_device_error() == M.MINW_OK
    return out, acts


@pytest.mark.parametrize("n,bits,hw,B", [(1, 3, 32, 4), (1, 1, 16, 3), (3, 2, 32, 2)])
def test_wresnet_stagewise(dev, M, n, bits, hw, B):
    """ResNet-8 and ResNet-20 shapes: every stage against the oracle."""
    net_p = wresnet_params(71 + n + bits, n=n, bits_w=bits, classes=10, hw=hw)
    x = wresnet_input(72 + n, B, hw=hw)
    logits, acts = _run(dev, M, net_p, x)
    st = net_p["stem"]
    stem = O.hardtanh(O.affine(O.conv2d_f32_seq(x, st["w"], 1, 1), st["scale"], st["shift"]))
    assert np.array_equal(acts[0], stem)
    thr = net_p["thr_w"]
    for i, blk in enumerate(net_p["blocks"]):
        _check_block(blk, acts[i], acts[i + 1], bits, thr)
    assert np.array_equal(logits, N.wresnet_head(net_p, acts[-1]))


def test_wresnet110_stagewise_sampled(dev, M):
    """ResNet-110 (n = 18, 54 blocks, 3-bit weights) at batch 16: all 16
    images through the GPU, images 0, 7 and 15 stage by stage against the
    oracle (each block recomputed from the GPU's input to it), and the head
    of every image."""
    B = 16
    net_p = wresnet_params(110, n=18, bits_w=3, classes=10, hw=32)
    x = wresnet_input(111, B, hw=32)
    logits, acts = _run(dev, M, net_p, x)
    pick = [0, 7, 15]
    st = net_p["stem"]
    stem = O.hardtanh(O.affine(O.conv2d_f32_seq(x[pick], st["w"], 1, 1), st["scale"], st["shift"]))
    assert np.array_equal(acts[0][pick], stem)
    thr = net_p["thr_w"]
    for i, blk in enumerate(net_p["blocks"]):
        _check_block(blk, acts[i][pick], acts[i + 1][pick], 3, thr)
    assert np.array_equal(logits, N.wresnet_head(net_p, acts[-1]))


def test_wresnet_without_kept_activations(dev, M):
    """The net without kept activations (ping-pong buffers) gives the same
    logits bit for bit, twice in a row (graph replay), and refuses the
    activation query."""
    net_p = wresnet_params(73, n=2, bits_w=3, classes=10, hw=32)
    x = wresnet_input(74, 5, hw=32)
    kept, _ = _run(dev, M, net_p, x, keep=True)
    net = M.Net.wresnet(net_p, 5, dev)
    logits = torch.empty((5, 10), dtype=torch.float32, device=dev)
    xt = dev_tensor(x, dev)
    outs = []
    for _ in range(2):
        net.forward(xt, logits)
        torch.cuda.synchronize()
        outs.append(logits.cpu().numpy())
    with pytest.raises(M.MinwError):
        net.wresnet_activation(0, torch.empty(5 * 16 * 32 * 32, device=dev))
    net.close()
    assert np.array_equal(outs[0], kept) and np.array_equal(outs[1], kept)
