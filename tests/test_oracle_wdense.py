"""Pin of the oracle's weight-only DenseNet-BC (Table III's DenseNet-100 with
3-bit weights and full-precision activations): every layer and transition of
a small net against a float64 torch restatement of the same wiring, fed the
oracle's own block features, the 2x2 average pool against numpy's mean, and
the head against numpy."""
import numpy as np
import pytest

from oracle import network as N
from paper_2003_04296_gb300.inputs import DEFAULT_THR, wdense_params, wresnet_input


def _levels(w, bits, thr):
    m = np.abs(w)
    s = np.where(w > 0, 1.0, -1.0)
    if bits == 1:
        return s
    if bits == 2:
        return np.where(m <= thr[0], 0.0, s)
    return 4.0 * np.where(m <= thr[2], 0.0, np.where(m <= thr[1], 0.25 * s, np.where(m <= thr[0], 0.5 * s, s)))


def test_avgpool2_against_numpy():
    t = np.random.default_rng(3).standard_normal((2, 3, 6, 8)).astype(np.float32)
    ref = t.astype(np.float64).reshape(2, 3, 3, 2, 4, 2).mean(axis=(3, 5))
    assert np.max(np.abs(N.avgpool2_f32(t) - ref)) < 4e-7


@pytest.mark.parametrize("bits", [3, 2])
def test_small_wdense(bits):
    torch = pytest.importorskip("torch")
    F_ = torch.nn.functional
    net = wdense_params(23, layers=3, growth=12, bits_w=bits, classes=10, hw=16)
    x = wresnet_input(24, 2, hw=16)
    logits, finals = N.wdense_forward(net, x, keep=True)
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    bf = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    thr = DEFAULT_THR[bits]
    wq = lambda c: _levels(c["w"] * c["w_scale"].reshape(-1, 1, 1, 1), bits, thr)
    bn = lambda y, c: y * c["scale"].reshape(1, -1, 1, 1) + c["shift"].reshape(1, -1, 1, 1)
    # stem, in fp64: the oracle's fp32 chain stays within a summation bound (then one bf16 rounding)
    st = net["stem"]
    stem = np.clip(bn(F_.conv2d(t(x), t(st["w"]), padding=1).numpy(), st), -1, 1)
    c0 = stem.shape[1]
    assert np.max(np.abs(finals[0][:, :c0] - stem)) <= 2.0 ** -7 + 1e-4
    c = c0
    for bi, lay_list in enumerate(net["blocks"]):
        Fb = finals[bi]
        for lay in lay_list:
            Fin = Fb[:, :c]
            h = np.clip(bn(F_.conv2d(t(Fin), t(wq(lay["b"]))).numpy(), lay["b"]), -1, 1)
            n = np.clip(bn(F_.conv2d(t(bf(h)), t(wq(lay["c"])), padding=1).numpy(), lay["c"]), -1, 1)
            err = np.abs(Fb[:, c:c + 12] - n)
            # the oracle stores bf16(n); fp32 roundings and bf16 flips of h stay far below a wiring error
            assert np.quantile(err, 0.99) <= 2.0 ** -8 + 1e-3 and np.max(err) < 0.1, f"block {bi} layer at {c}"
            c += 12
        assert Fb.shape[1] == c
        if bi < 2:
            tr = net["trans"][bi]
            tt = np.clip(bn(F_.conv2d(t(Fb), t(wq(tr))).numpy(), tr), -1, 1)
            ref = tt.reshape(tt.shape[0], tt.shape[1], tt.shape[2] // 2, 2, tt.shape[3] // 2, 2).mean(axis=(3, 5))
            nxt = finals[bi + 1][:, :c // 2]
            err = np.abs(nxt - ref)
            assert np.quantile(err, 0.99) <= 2.0 ** -8 + 1e-3 and np.max(err) < 0.1
            c //= 2
    fc = net["fc"]
    pooled = finals[-1].astype(np.float64).mean(axis=(2, 3))
    ref = (pooled @ fc["w"].astype(np.float64).T) * fc["scale"] + fc["shift"]
    assert np.max(np.abs(logits - ref)) < 1e-4 * (1 + np.max(np.abs(ref)))
