"""GPU parity of the whole-network forward (minw_forward) against the oracle:
a small Model-A-shaped ConvNet for every activation/weight bit pair the
workloads use, and the full CIFAR ConvNet at batch 256 on sampled images."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from paper_2003_04296_gb300.inputs import convnet_input, convnet_params  # noqa: E402
from tests._gpu import assert_close, dev_tensor  # noqa: E402

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


def _run(dev, M, net_p, x_np, variant):
    net = M.Net(M.layer_descs(net_p, dev), max_batch=x_np.shape[0], variant=variant)
    logits = torch.empty((x_np.shape[0], net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x_np, dev), logits)
    torch.cuda.synchronize()
    out = logits.cpu().numpy()
    net.close()
    return out


@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 1), (2, 2), (3, 3)])
def test_small_convnet(dev, M, bits_a, bits_w):
    net_p = convnet_params(41, bits_a=bits_a, bits_w=bits_w, widths=(64, 64, 128, 128),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(42, 3, hw=16)
    got = _run(dev, M, net_p, x, M.VARIANT_POPC)
    ref = N.convnet_forward(net_p, x)
    assert_close(got, ref)
    assert np.array_equal(got, ref)     # same fp32 operations in the same order


@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 2), (3, 3)])
def test_small_convnet_tensor_cores(dev, M, bits_a, bits_w):
    """Widths that are multiples of 128 put every quantized layer on the
    tensor-core path (codes layout between layers)."""
    net_p = convnet_params(43, bits_a=bits_a, bits_w=bits_w, widths=(128, 128, 256, 256),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(44, 5, hw=16)
    got = _run(dev, M, net_p, x, M.VARIANT_AUTO)
    ref = N.convnet_forward(net_p, x)
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("model", ["B", "C", "D"])
@pytest.mark.parametrize("bits_a,bits_w", [(1, 1), (2, 1)])
def test_cifar_models_b_to_d(dev, M, model, bits_a, bits_w):
    """Models B-D of Sec. IV-B (Model A with half the convolution channels,
    then half the hidden FC units, twice) at 32 x 32, batch 20, against the
    oracle's logits bit for bit."""
    from paper_2003_04296_gb300.inputs import CIFAR_MODELS
    net_p = convnet_params(60 + ord(model), bits_a=bits_a, bits_w=bits_w, **CIFAR_MODELS[model])
    x = convnet_input(61 + ord(model), 20)
    got = _run(dev, M, net_p, x, M.VARIANT_AUTO)
    ref = N.convnet_forward(net_p, x)
    assert np.array_equal(got, ref)


def test_cifar_convnet_batch256_sampled(dev, M):
    """The full Model-A-shaped ConvNet (128-128-P-256-256-P-512-512-P,
    FC 1024-1024-10), 1-bit, batch 256: 16 images spread over the batch (every
    wave of tiles, the last one included) re-run by the oracle, bit for bit."""
    from tests import _oracle_pool as OP
    net_p = convnet_params(2, bits_a=1, bits_w=1)
    x = convnet_input(2, 256)
    got = _run(dev, M, net_p, x, M.VARIANT_AUTO)
    assert np.all(np.isfinite(got))
    idx = OP.spread(256)
    refs = OP.starmap(OP.convnet_logits, [(2, 1, 1, 2, 256, i) for i in idx])
    for i, ref in zip(idx, refs):
        assert np.array_equal(got[i:i + 1], ref), f"image {i}"


@pytest.mark.parametrize("batch,bits", [(64, 1), (2, 2)])
def test_auto_choice_is_the_measured_fastest(dev, M, batch, bits):
    """MINW_VARIANT_AUTO times every layer the tensor cores cover on each
    candidate (E4M3, E2M1, E2M1 CTA pairs, popcount on bit-planes) at creation
    and keeps the fastest: the kernel each layer reports is the least of its
    measured times, the popcount path was measured for every such layer, and
    the net (whatever mix of layouts the measurement produced) still gives the
    oracle's logits bit for bit.  Batch 2 makes the tensor-core tiles mostly
    empty, where the popcount path can win."""
    net_p = convnet_params(47, bits_a=bits, bits_w=bits, widths=(64, 128, 128, 256),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(48, batch, hw=16)
    net = M.Net(M.layer_descs(net_p, dev), max_batch=batch, variant=M.VARIANT_AUTO)
    variants = net.layer_variants()
    kind = {M.VARIANT_TC: 0, M.VARIANT_TC_E2M1: 1, M.VARIANT_TC_E2M1_PAIRS: 2, M.VARIANT_POPC: 3,
            M.VARIANT_TC_E2M1_N128: 4}
    assert net.layer_candidates(0) == [-1.0] * 5
    for layer in range(1, net.launches):
        ms = net.layer_candidates(layer)
        assert ms[0] > 0 and ms[3] > 0, (layer, ms)      # E4M3 and popcount cover every layer here
        measured = [t if t >= 0 else np.inf for t in ms]
        assert kind[variants[layer]] == int(np.argmin(measured)), (layer, variants[layer], ms)
    logits = torch.empty((batch, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    got = logits.cpu().numpy()
    net.close()
    assert np.array_equal(got, N.convnet_forward(net_p, x))


def test_per_layer_requests_replay_a_plan(dev, M):
    """A per-layer kernel request (minw_layer_desc.variant) skips that layer's
    measurement and runs the requested kernel: popcount, E4M3, E2M1 CTA pairs
    and E2M1 single-CTA 128-channel tiles mixed in one net (each layer's input layout follows its
    consumer), requested in the values minw_net_layer_variants reports
    (VARIANT_TC: E4M3 operands) and reported back unchanged, with the oracle's
    logits bit for bit."""
    net_p = convnet_params(49, bits_a=2, bits_w=1, widths=(128, 128, 256, 256),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(50, 24, hw=16)
    req = [0, M.VARIANT_POPC, M.VARIANT_TC, M.VARIANT_TC_E2M1_PAIRS, M.VARIANT_TC_E2M1_N128, M.VARIANT_POPC]
    descs = M.layer_descs(net_p, dev)
    assert len(descs) == len(req)
    for d, v in zip(descs, req):
        d["variant"] = v
    net = M.Net(descs, max_batch=24, variant=M.VARIANT_AUTO)
    assert net.layer_variants() == req
    for layer in range(net.launches):
        assert net.layer_candidates(layer) == [-1.0] * 5        # nothing measured
    logits = torch.empty((24, net.out_features), dtype=torch.float32, device=dev)
    net.forward(dev_tensor(x, dev), logits)
    torch.cuda.synchronize()
    got = logits.cpu().numpy()
    net.close()
    assert np.array_equal(got, N.convnet_forward(net_p, x))
