"""The plan options (minw_set_plan_options) and the bounded-wait timeout path,
on the GPU through the C ABI.

Every option picks between kernel variants that compute the same results, so
each one turned off (or set to its other value) must leave a network's logits
equal to the oracle's bit for bit.  The timeout path is exercised without any
fault: minw_test_stall_next_launch makes the next launch wait on a barrier that
nothing completes; with a short wait limit that wait runs out, the kernel
winds down, minw_get_last_device_error reports MINW_ETIMEOUT once, and the next
normal call is correct and reports MINW_OK."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import network as N  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem, convnet_input, convnet_params  # noqa: E402
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


@pytest.fixture
def restore(M):
    yield
    M.set_plan_options()
    M.minw_test_stall_next_launch(0)


def _net_logits(dev, M, net_p, x, variant=0, host=False):
    net = M.Net(M.layer_descs(net_p, dev), max_batch=x.shape[0], variant=variant)
    if host:
        out = np.empty((x.shape[0], net.out_features), dtype=np.float32)
        net.forward_host(np.ascontiguousarray(x), out)
    else:
        logits = torch.empty((x.shape[0], net.out_features), dtype=torch.float32, device=dev)
        xd = dev_tensor(x, dev)
        net.forward(xd, logits)
        net.forward(xd, logits)          # the second call replays the captured graph (when on)
        torch.cuda.synchronize()
        out = logits.cpu().numpy()
    net.close()
    return out


OPTION_CASES = [
    dict(cta_pairs=0),
    dict(channel_major=0),
    dict(channel_major_min_tiles_per_sm=0),      # channel-major tiles even for a small batch
    dict(channel_major_min_tiles_per_sm=0, dup_weights=0),
    dict(kblocks_per_stage=1),
    dict(tma_lanes=1),
    dict(tma_lanes=8),
    dict(resident_weights=1),
    dict(resident_weights=1, tma_lanes=2),
    dict(first_tma=0),
    dict(first_tensor_cores=0),
    dict(first_tensor_cores=0, first_tma=0),
    dict(pdl=0),
    dict(graph=0),
]


@pytest.mark.parametrize("opts", OPTION_CASES, ids=lambda d: ",".join(f"{k}={v}" for k, v in d.items()))
@pytest.mark.parametrize("variant", [0, 3])
def test_options_keep_the_logits(dev, M, restore, opts, variant):
    """A small ConvNet (64- to 512-channel layers, pooled, fully connected
    head) under each option, on E2M1 (auto) and E4M3 operands."""
    net_p = convnet_params(61, bits_a=2, bits_w=2, widths=(64, 128, 256, 512),
                           pools=(False, True, False, True), fcs=(256,), classes=10, hw=16)
    x = convnet_input(62, 6, hw=16)
    ref = N.convnet_forward(net_p, x)
    M.set_plan_options(**opts)
    got = _net_logits(dev, M, net_p, x, variant=variant)
    assert np.array_equal(got, ref)
    assert M.minw_get_last_device_error() == M.MINW_OK


def test_options_round_trip_and_validation(M, restore):
    d = M.get_plan_options()
    assert d["cta_pairs"] == 1 and d["kblocks_per_stage"] == 2 and d["tma_lanes"] == 1 and d["wait_cycles"] == 1 << 31
    M.set_plan_options(kblocks_per_stage=1, wait_cycles=12345)
    got = M.get_plan_options()
    assert got["kblocks_per_stage"] == 1 and got["wait_cycles"] == 12345
    with pytest.raises(M.MinwError):
        M.set_plan_options(kblocks_per_stage=3)
    with pytest.raises(M.MinwError):
        M.set_plan_options(wait_cycles=0)
    with pytest.raises(M.MinwError):
        M.set_plan_options(tma_lanes=9)
    M.set_plan_options()
    assert M.get_plan_options() == d


def _small_block(dev, M, seed):
    p = conv_problem(seed, 2, 128, 8, 8, 64, 3, 3, 1, 1, 1, 1, w_sigma=0.5)
    act = torch.empty((2, 8, 8, 128), dtype=torch.uint8, device=dev)
    wgt = torch.empty((64, 3, 3, 128), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(1, p["thr_a"]), act)
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(1, p["thr_w"]), wgt,
                             channel_scale=dev_tensor(p["w_scale"], dev))
    al = O.quantize(p["x"], 1, p["thr_a"])
    wl = O.quantize(p["w"], 1, p["thr_w"], p["w_scale"])
    return p, act, wgt, O.conv2d_levels(al, wl, 1, 1, 1, 1)


def test_timeout_tensor_core_kernel(dev, M, restore):
    """The single-CTA tensor-core kernel with a stalled MMA issuer: every wait
    runs out within the short limit, MINW_ETIMEOUT is reported once, and the
    next launch (no stall) gives the exact accumulators and MINW_OK."""
    assert M.minw_get_last_device_error() == M.MINW_OK
    p, act, wgt, ref = _small_block(dev, M, 5)
    M.set_plan_options(wait_cycles=1 << 20)
    acc = torch.full((2, 64, 8, 8), -7, dtype=torch.int32, device=dev)
    M.minw_test_stall_next_launch(M.STALL_CONV_TC)
    M.minw_conv2d_codes(act, 2, 128, 8, 8, 1, wgt, 64, 3, 3, 1, 1, 1, acc_out=acc)
    assert M.minw_get_last_device_error() == M.MINW_ETIMEOUT
    assert M.minw_get_last_device_error() == M.MINW_OK          # read once, then cleared
    M.minw_conv2d_codes(act, 2, 128, 8, 8, 1, wgt, 64, 3, 3, 1, 1, 1, acc_out=acc)
    assert M.minw_get_last_device_error() == M.MINW_OK
    assert np.array_equal(acc.cpu().numpy(), ref)


def test_timeout_first_layer(dev, M, restore):
    """The fp32 first layer (TMA patches) with a stalled start: MINW_ETIMEOUT
    once, the in-flight patches drained, then a correct run and MINW_OK."""
    assert M.minw_get_last_device_error() == M.MINW_OK
    r = np.random.default_rng(8)
    x = r.uniform(-1, 1, (3, 3, 16, 16)).astype(np.float32)
    w = r.normal(0, 0.05, (64, 3, 3, 3)).astype(np.float32)
    sc = np.abs(r.normal(1, 0.1, 64)).astype(np.float32)
    sh = r.normal(0, 0.1, 64).astype(np.float32)
    xd, wd, scd, shd = (dev_tensor(a, dev) for a in (x, w, sc, sh))
    y = torch.empty((3, 64, 16, 16), dtype=torch.float32, device=dev)
    M.set_plan_options(wait_cycles=1 << 20)
    M.minw_test_stall_next_launch(M.STALL_CONV_FIRST)
    M.minw_conv_first(xd, wd, 1, 1, scd, shd, q_w=M.quant(1, DEFAULT_THR[1]), y_out=y)
    assert M.minw_get_last_device_error() == M.MINW_ETIMEOUT
    M.minw_conv_first(xd, wd, 1, 1, scd, shd, q_w=M.quant(1, DEFAULT_THR[1]), y_out=y)
    assert M.minw_get_last_device_error() == M.MINW_OK
    wl = O.quantize(w, 1, DEFAULT_THR[1])
    assert np.array_equal(y.cpu().numpy(), O.affine(O.conv2d_f32_seq(x, wl, 1, 1), sc, sh))
