"""Host logic of bench.py's weight-only network workloads (no GPU): the
per-op MAC lists follow the networks' timed-op order (the order
minw_net_layer_times reports: ResNet-110's stem, its pass, per block conv1,
[the 1x1 / 2 shortcut], conv2, then the head; DenseNet-100's stem, its pass,
per layer the 1x1 and the 3x3, per transition its convolution and pool, then
the head), the roofline's convolution indices pick exactly the
tensor-core convolutions, and their MACs add up to the networks' own
unpadded counts."""
import types

import bench


def _wl(name):
    return bench.Workload(name, types.SimpleNamespace(bits_a=1, bits_w=1, bits_a_resnet=3, bits_w_resnet=3))


def test_wresnet110_op_list():
    wl = _wl("wresnet110")
    macs, q = wl.op_macs()
    P = wl.params
    assert len(macs) == 3 + sum(3 if b["down"] is not None else 2 for b in P["blocks"]) == 113
    assert len(q) == 110 and all(macs[i] > 0 for i in q)
    assert macs[1] == 0 and set(range(2, len(macs) - 1)) == set(q)
    want, hw, c = 0, P["hw"], 16
    for b in P["blocks"]:
        o = b["c1"]["w"].shape[0]
        hw //= b["stride"]
        want += hw * hw * o * (c * 9 + o * 9 + (c if b["down"] is not None else 0))
        c = o
    assert sum(macs[i] for i in q) == want


def test_densenet100_op_list():
    wl = _wl("wdense100")
    macs, q = wl.op_macs()
    P = wl.params
    L, k = P["layers"], P["growth"]
    assert len(macs) == 2 + 2 * 3 * L + 2 * 2 + 1 == 103
    assert len(q) == 3 * 2 * L + 2 and all(macs[i] > 0 for i in q)
    pools = [i for i in range(2, len(macs) - 1) if i not in q]
    assert len(pools) == 2 and all(macs[i] == 0 for i in pools)
    # 96 layer convolutions and two transitions, unpadded: channels 24 + 12 i in block 1, ...
    want, c = 0, 2 * k
    for b in range(3):
        px = (P["hw"] >> b) ** 2
        for i in range(L):
            want += px * (4 * k * c + k * 4 * k * 9)
            c += k
        if b < 2:
            want += px * (c // 2) * c
            c //= 2
    assert sum(macs[i] for i in q) == want
    assert P["features"] == c == 342


def test_weight_only_configs_name_their_workloads():
    for name, tag in (("wresnet110", "wresnet110_cifar_fwd_w3"), ("wdense100", "densenet100_bc_k12_cifar_fwd_w3")):
        cfg = _wl(name).config(1)
        assert cfg["workload"] == tag and cfg["batch_per_gpu"] == 128 and cfg["bits_w"] == 3
