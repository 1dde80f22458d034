"""GPU parity of the ResNet-18-shaped forward (minw_resnet18_create +
minw_forward) against the oracle: small images for every bit width (the last
stages run at 1x1 and 2x2 spatial sizes, where split-K engages), and the
ImageNet-shaped workload (batch 128, 224x224, 3-bit) on sampled images."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from paper_2003_04296_gb300.inputs import resnet18_input, resnet18_params  # noqa: E402
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


def _forward(M, dev, params, x_np):
    net = M.Net.resnet18(params, max_batch=x_np.shape[0], device=dev)
    logits = torch.empty((x_np.shape[0], params["classes"]), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x_np, dev), logits)
    torch.cuda.synchronize()
    assert M.minw_get_last_device_error() == M.MINW_OK
    out = logits.cpu().numpy()
    return net, out


@pytest.mark.parametrize("bits", [3, 2, 1])
@pytest.mark.parametrize("hw,B", [(32, 3), (64, 2)])
def test_small_resnet(dev, M, bits, hw, B):
    params = resnet18_params(61 + bits, bits_a=bits, bits_w=bits, classes=37, hw=hw)
    x = resnet18_input(62 + hw, B, hw=hw)
    net, got = _forward(M, dev, params, x)
    assert net.launches == 3 + 8 * 2 + 3
    net.close()
    ref = N.resnet18_forward(params, x)
    assert np.array_equal(got, ref)     # same fp32 operations in the same order


def test_resnet_host_buffers(dev, M):
    params = resnet18_params(71, classes=16, hw=32)
    x = resnet18_input(72, 4, hw=32)
    net, got = _forward(M, dev, params, x)
    out = np.empty((4, 16), dtype=np.float32)
    net.forward_host(x, out)
    net.close()
    assert np.array_equal(out, got)


def test_resnet_timing_and_variants(dev, M):
    params = resnet18_params(73, classes=8, hw=32)
    x = resnet18_input(74, 2, hw=32)
    net = M.Net.resnet18(params, max_batch=2, device=dev)
    net.enable_timing(True)
    logits = torch.empty((2, 8), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    ms = net.layer_times()
    var = net.layer_variants()
    net.close()
    assert len(ms) == len(var) == 22 and all(t >= 0.0 for t in ms)
    # block convolutions in forward order (conv1, [shortcut], conv2): inputs of
    # 128 channels or more are E2M1 codes, the 64-channel ones E4M3
    c_in = [64, 64, 64, 64, 64, 64, 128, 128, 128, 128, 128, 256, 256, 256, 256, 256, 512, 512, 512]
    want = [M.VARIANT_TC_E2M1 if c % 128 == 0 else M.VARIANT_TC for c in c_in]
    assert var[0] == 0 and var[1] == 0 and var[-1] == 0 and var[2:-1] == want


def test_resnet_create_errors(dev, M):
    params = resnet18_params(75, classes=8, hw=32)
    bad = dict(params, hw=48)              # not a multiple of 32
    with pytest.raises(M.MinwError):
        M.Net.resnet18(bad, max_batch=2, device=dev)


def test_resnet18_imagenet_b128_sampled(dev, M):
    """The ImageNet-shaped workload: batch 128 of 224x224 images, 3-bit
    activations and weights, 1000 classes; images are independent, so the
    oracle checks 16 of them spread over the batch (every wave of tiles of
    every layer, the last one included) bit for bit."""
    from tests import _oracle_pool as OP
    params = resnet18_params(0, bits_a=3, bits_w=3, classes=1000, hw=224)
    x = resnet18_input(1, 128, hw=224)
    net, got = _forward(M, dev, params, x)
    net.close()
    assert np.all(np.isfinite(got))
    idx = OP.spread(128)
    refs = OP.starmap(OP.resnet_logits, [(0, 3, 3, 1000, 224, 1, 128, i) for i in idx])
    for i, ref in zip(idx, refs):
        assert np.array_equal(got[i:i + 1], ref), f"image {i}"
