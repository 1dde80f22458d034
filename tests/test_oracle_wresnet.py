"""Pin of the oracle's weight-only residual network (Table III's ResNet-(6n+2)
with 3-bit weights and full-precision activations): every block of a small
net against a float64 torch restatement of the same wiring, fed the oracle's
own block input, and the head against numpy."""
import numpy as np
import pytest

from oracle import network as N
from paper_2003_04296_gb300.inputs import DEFAULT_THR, wresnet_input, wresnet_params


def _levels(w, bits, thr):
    """Weight levels in integer units, from Eq. qnn's thresholds as written
    (an independent restatement of the quantizer for the composition pin)."""
    m = np.abs(w)
    s = np.where(w > 0, 1.0, -1.0)
    if bits == 1:
        return np.where(w > 0, 1.0, -1.0)
    if bits == 2:
        return np.where(m <= thr[0], 0.0, s)
    return 4.0 * np.where(m <= thr[2], 0.0, np.where(m <= thr[1], 0.25 * s, np.where(m <= thr[0], 0.5 * s, s)))


@pytest.mark.parametrize("bits", [3, 1])
def test_small_wresnet_blocks(bits):
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    net = wresnet_params(19, n=1, bits_w=bits, classes=10, hw=16)
    x = wresnet_input(20, 2, hw=16)
    logits, trace = N.wresnet_forward(net, x, keep=True)
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    bf = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16).to(torch.float64)
    # stem in fp64: the oracle's fp32 fmaf chain stays within a summation bound
    st = net["stem"]
    z = F.conv2d(t(x), t(st["w"]), padding=1).numpy()
    ref = np.clip(z * st["scale"].reshape(1, -1, 1, 1) + st["shift"].reshape(1, -1, 1, 1), -1, 1)
    assert np.max(np.abs(trace[0] - ref)) < 1e-4
    thr = DEFAULT_THR[bits]
    for i, blk in enumerate(net["blocks"]):
        a = trace[i]
        wq = lambda c: _levels(c["w"] * c["w_scale"].reshape(-1, 1, 1, 1), bits, thr)
        c1, c2 = blk["c1"], blk["c2"]
        y1 = F.conv2d(bf(a), t(wq(c1)), stride=blk["stride"], padding=1).numpy()
        h = np.clip(y1 * c1["scale"].reshape(1, -1, 1, 1) + c1["shift"].reshape(1, -1, 1, 1), -1, 1)
        y2 = F.conv2d(bf(h), t(wq(c2)), padding=1).numpy()
        y2 = y2 * c2["scale"].reshape(1, -1, 1, 1) + c2["shift"].reshape(1, -1, 1, 1)
        if blk["down"] is None:
            s = a.astype(np.float64)
        else:
            d = blk["down"]
            s = F.conv2d(bf(a), t(wq(d)), stride=2).numpy()
            s = s * d["scale"].reshape(1, -1, 1, 1) + d["shift"].reshape(1, -1, 1, 1)
        ref = np.clip(y2 + s, -1, 1)
        # fp32 roundings and the bf16 rounding of h (which can land on the other side of a
        # rounding boundary than the fp64 restatement's) move outputs by far less than a wrong
        # wiring, tap, stride or shortcut would
        err = np.abs(trace[i + 1] - ref)
        assert np.quantile(err, 0.99) < 1e-3, f"block {i}: 99th percentile {np.quantile(err, 0.99):.2e}"
        assert np.max(err) < 0.1
    fc = net["fc"]
    pooled = trace[-1].astype(np.float64).mean(axis=(2, 3))
    ref = (pooled @ fc["w"].astype(np.float64).T) * fc["scale"] + fc["shift"]
    assert np.max(np.abs(logits - ref)) < 1e-4 * (1 + np.max(np.abs(ref)))
