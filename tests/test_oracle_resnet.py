"""Pin of the oracle's ResNet-18 composition (stem, residual blocks, head)
against a float64 torch restatement of the same wiring on a small input."""
import numpy as np
import pytest

from oracle import network as N
from paper_2003_04296_gb300.inputs import DEFAULT_THR, resnet18_input, resnet18_params


def _levels(y, bits, thr):
    if bits == 1:
        return np.where(y > 0, 1.0, -1.0)
    m = np.abs(y)
    s = np.where(y > 0, 1.0, -1.0)
    if bits == 2:
        return np.where(m <= thr[0], 0.0, s)
    return np.where(m <= thr[2], 0.0, np.where(m <= thr[1], 0.25 * s, np.where(m <= thr[0], 0.5 * s, s)))


@pytest.mark.parametrize("bits", [3, 1])
def test_small_resnet_blocks(bits):
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    net = resnet18_params(9, bits_a=bits, bits_w=bits, classes=10, hw=32)
    x = resnet18_input(10, 2, hw=32)
    logits, trace = N.resnet18_forward(net, x, keep=True)
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    # stem, in fp64: the oracle's fp32 fmaf chain stays within a summation bound
    st = net["stem"]
    z = F.max_pool2d(F.conv2d(t(x), t(st["w"]), stride=2, padding=3), 3, 2, 1).numpy()
    ref = np.clip(z * st["scale"].reshape(1, -1, 1, 1) + st["shift"].reshape(1, -1, 1, 1), -1, 1)
    assert np.max(np.abs(trace[0] - ref)) < 1e-4
    thr = DEFAULT_THR[bits]
    for i, blk in enumerate(net["blocks"]):
        a = trace[i]
        u = _levels(a, bits, thr)
        wq = lambda c: _levels(c["w"] * c["w_scale"].reshape(-1, 1, 1, 1), bits, thr)
        c1, c2 = blk["c1"], blk["c2"]
        y1 = F.conv2d(t(u), t(wq(c1)), stride=blk["stride"], padding=1).numpy()
        y1 = np.clip(y1 * (2 ** (4 if bits == 3 else 0)) * c1["scale"].reshape(1, -1, 1, 1)
                     + c1["shift"].reshape(1, -1, 1, 1), -1, 1)
        v = _levels(y1.astype(np.float32), bits, thr)
        y2 = F.conv2d(t(v), t(wq(c2)), padding=1).numpy() * (2 ** (4 if bits == 3 else 0))
        y2 = y2 * c2["scale"].reshape(1, -1, 1, 1) + c2["shift"].reshape(1, -1, 1, 1)
        if blk["down"] is None:
            s = u
        else:
            d = blk["down"]
            s = F.conv2d(t(u), t(wq(d)), stride=2).numpy() * (2 ** (4 if bits == 3 else 0))
            s = s * d["scale"].reshape(1, -1, 1, 1) + d["shift"].reshape(1, -1, 1, 1)
        ref = np.clip(y2 + s, -1, 1)
        # block outputs agree except where an fp32 rounding flips a level upstream
        close = np.abs(trace[i + 1] - ref) <= 1e-5 + 1e-5 * np.abs(ref)
        assert close.mean() > 0.999, f"block {i}: {1 - close.mean():.2e} of outputs differ"
    assert logits.shape == (2, 10) and np.all(np.isfinite(logits))
