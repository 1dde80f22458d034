"""minw_fc_codes_noalloc: the fully connected layer for callers that cannot
allocate device memory (a plugin inside a framework that owns all device
memory, a service that forbids allocations after start-up).  Its split-K
scratch is a fixed array inside the library.

Checked through the C ABI against minw_fc_codes with a caller-allocated
workspace, on two calls in a row, at the tolerance of the other GPU tests
(exact integers and codes, fp32 within 1e-5 relative / 1e-6 absolute), and
against the oracle itself (exact accumulators, the BN output and the next
layer's levels bit for bit).
This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes on its own in a fresh process."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem  # noqa: E402
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


def _operands(dev, M, B, K, Oc, ba, bw, seed):
    p = conv_problem(seed, B, K, 1, 1, Oc, 1, 1, 1, 0, ba, bw, w_sigma=0.5)
    act = torch.empty((B, K), dtype=torch.uint8, device=dev)
    wgt = torch.empty((Oc, K), dtype=torch.uint8, device=dev)
    M.aqe_quantize_codes(dev_tensor(p["x"], dev), M.quant(ba, p["thr_a"]), act.view(B, 1, 1, K))
    M.minw_pack_weight_codes(dev_tensor(p["w"], dev), M.quant(bw, p["thr_w"]), wgt.view(Oc, 1, 1, K),
                             channel_scale=dev_tensor(p["w_scale"], dev))
    return p, act, wgt


def _outputs(dev, B, Oc, last):
    acc = torch.full((B, Oc), -7, dtype=torch.int32, device=dev)
    y = torch.full((B, Oc), float("nan"), dtype=torch.float32, device=dev)
    codes = None if last else torch.full((B, Oc), 0x77, dtype=torch.uint8, device=dev)
    return acc, y, codes


def _decode_e4m3(b):
    """E4M3 bytes to values from the format's definition (normal numbers and 0)."""
    b = b.astype(np.int64)
    v = np.where(b & 0x80, -1.0, 1.0) * (1.0 + (b & 7) / 8.0) * np.power(2.0, ((b >> 3) & 0xF) - 7.0)
    return np.where((b & 0x7F) == 0, 0.0, v)


@pytest.mark.parametrize("B,K,Oc,ba,bw", [(256, 8192, 1024, 1, 1), (64, 4096, 512, 3, 3), (256, 2048, 10, 1, 1)])
def test_noalloc_matches_workspace_entry_point(dev, M, B, K, Oc, ba, bw):
    p, act, wgt = _operands(dev, M, B, K, Oc, ba, bw, seed=B + K + Oc)
    # the fixed array really carries a split of K for the shapes that split
    if Oc >= 512:
        assert M.minw_fc_ksplit(B, K, Oc, 8 << 20) > 1
    sc, sh = dev_tensor(p["scale"], dev), dev_tensor(p["shift"], dev)
    last = Oc % 16 != 0
    q = None if last else M.quant(ba, DEFAULT_THR[ba])

    # reference: the existing entry point with a caller-allocated workspace
    ws = torch.empty(max(M.minw_fc_workspace_bytes(B, K, Oc), 16), dtype=torch.uint8, device=dev)
    acc_r, y_r, codes_r = _outputs(dev, B, Oc, last)
    M.minw_fc_codes(act, B, K, ba, wgt, Oc, bw, scale=sc, shift=sh, q_out=q, codes_out=codes_r, y_out=y_r,
                    acc_out=acc_r, workspace=ws)
    torch.cuda.synchronize()

    free_after_first = None
    for call in range(2):
        acc, y, codes = _outputs(dev, B, Oc, last)
        torch.cuda.synchronize()
        if call == 1:
            free_after_first = torch.cuda.mem_get_info()[0]
        M.minw_fc_codes_noalloc(act, B, K, ba, wgt, Oc, bw, scale=sc, shift=sh, q_out=q, codes_out=codes,
                                y_out=y, acc_out=acc)
        torch.cuda.synchronize()
        if call == 1:
            assert torch.cuda.mem_get_info()[0] == free_after_first, "the call allocated device memory"
        assert np.array_equal(acc.cpu().numpy(), acc_r.cpu().numpy())
        assert_close(y.cpu().numpy(), y_r.cpu().numpy())
        if codes is not None:
            assert np.array_equal(codes.cpu().numpy(), codes_r.cpu().numpy())
    assert M.minw_get_last_device_error() == M.MINW_OK

    # against the oracle: exact accumulators, BN (+ HardTanh), the next layer's levels
    al = O.quantize(p["x"], ba, p["thr_a"])
    wl = O.quantize(p["w"], bw, p["thr_w"], p["w_scale"])
    ref = O.conv2d_levels(al, wl, 1, 0, ba, bw).reshape(B, Oc)
    assert np.array_equal(acc.cpu().numpy(), ref)
    yref = O.affine(ref, p["scale"], p["shift"])
    if not last:
        yref = O.hardtanh(yref)
        lv = O.quantize(yref, ba, DEFAULT_THR[ba]) * 2.0 ** O.units_shift(ba)
        assert np.array_equal(_decode_e4m3(codes.cpu().numpy()), lv)
    assert np.array_equal(y.cpu().numpy(), yref)


def test_noalloc_rejects_requests_beyond_the_fixed_scratch(dev, M):
    """1024 x 2048 -> 1024 would split K into slices whose two smallest
    partial-sum buffers alone exceed the fixed array: rejected before any launch."""
    B, K, Oc = 1024, 2048, 1024
    act = torch.zeros((B, K), dtype=torch.uint8, device=dev)
    wgt = torch.zeros((Oc, K), dtype=torch.uint8, device=dev)
    acc = torch.zeros((B, Oc), dtype=torch.int32, device=dev)
    with pytest.raises(M.MinwError) as err:
        M.minw_fc_codes_noalloc(act, B, K, 1, wgt, Oc, 1, acc_out=acc)
    assert err.value.status == M.MINW_EUNSUPPORTED
