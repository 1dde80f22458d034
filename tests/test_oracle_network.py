"""Pin of the oracle's network composition (Algorithm 1 inference branch with
the layer constructs of Sec. III-E) against a float64 torch restatement of the
same block structure on a small Model-A-shaped ConvNet."""
import numpy as np
import pytest

from oracle import network as N
from paper_2003_04296_gb300.inputs import DEFAULT_THR, convnet_input, convnet_params


def _levels(y, bits, thr):
    """Level sets of Sec. IV-A, restated with numpy for this test."""
    if bits == 1:
        return np.where(y > 0, 1.0, -1.0)
    m = np.abs(y)
    s = np.where(y > 0, 1.0, -1.0)
    if bits == 2:
        return np.where(m <= thr[0], 0.0, s)
    return np.where(m <= thr[2], 0.0, np.where(m <= thr[1], 0.25 * s,
                    np.where(m <= thr[0], 0.5 * s, s)))


@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 1), (2, 2), (3, 3)])
def test_small_convnet_layerwise(bits_a, bits_w):
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    net = convnet_params(21, bits_a=bits_a, bits_w=bits_w, widths=(32, 32, 64, 64),
                         pools=(False, True, False, True), fcs=(64,), classes=10, hw=8)
    x = convnet_input(22, 2, hw=8)
    logits, trace = N.convnet_forward(net, x, keep=True)
    a = x
    for li, (layer, (acc, y)) in enumerate(zip(net["layers"], trace)):
        wl = _levels(layer["w"].astype(np.float32) * layer["w_scale"].reshape(-1, *([1] * (layer["w"].ndim - 1))),
                     layer["bits_w"], DEFAULT_THR[layer["bits_w"]])
        if li == 0:
            # fp32 first layer: compare against fp64 within a summation bound
            z = F.conv2d(torch.from_numpy(a).double(), torch.from_numpy(wl), padding=1).numpy()
            ref = z * layer["scale"].reshape(1, -1, 1, 1) + layer["shift"].reshape(1, -1, 1, 1)
            ref = np.clip(ref, -1, 1)
            assert np.max(np.abs(y - ref)) < 1e-4
        else:
            al = _levels(a, layer["bits_in"], DEFAULT_THR[layer["bits_in"]])
            u = 2 ** ((2 if layer["bits_in"] == 3 else 0) + (2 if layer["bits_w"] == 3 else 0))
            if layer["kind"] == "conv":
                z = F.conv2d(torch.from_numpy(al), torch.from_numpy(wl), padding=1)
                if layer["pool"]:
                    z = F.max_pool2d(z, 2, 2)
                z = z.numpy() * u
            else:
                z = (torch.from_numpy(al.reshape(al.shape[0], -1)) @ torch.from_numpy(wl).T).numpy() * u
            assert np.array_equal(acc, z.astype(np.int64))
            sh = (1, -1) + (1,) * (acc.ndim - 2)
            ref = acc.astype(np.float64) * layer["scale"].reshape(sh) + layer["shift"].reshape(sh)
            if layer["bits_out"]:
                ref = np.clip(ref, -1, 1)
            assert np.max(np.abs(y - ref)) <= 1e-6 * np.max(np.abs(ref)) + 1e-6
        a = y
    assert logits.shape == (2, 10)
    assert np.all(np.isfinite(logits))
