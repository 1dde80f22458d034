"""The C-ABI library loads, exports every entry point include/minw.h declares,
and rejects bad arguments on the host before touching a device (no GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "minw.h")).read()
    return sorted(set(re.findall(r"^MINW_API\s+[\w\s\*]*?\b(\w+)\s*\(", src, re.M)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g
    g.build()
    from paper_2003_04296_gb300 import minw
    return minw.lib()


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    from paper_2003_04296_gb300 import minw
    assert set(names) == set(minw.SIGNATURES)


def test_status_strings(lib):
    from paper_2003_04296_gb300 import minw
    assert minw.status_string(0) == "ok"
    assert "invalid" in minw.status_string(1)
    assert lib.minw_version() >= 100


def test_host_side_validation(lib):
    from paper_2003_04296_gb300 import minw
    q = minw.quant(1)
    P = ctypes.c_void_p
    fake = P(4096)                     # never dereferenced: validation fails first
    # negative length, bad bits, bad alpha
    assert lib.aqe_forward(fake, fake, -1, 0.5, ctypes.byref(q), None) == minw.MINW_EINVAL
    assert lib.aqe_forward(fake, fake, 0, 0.5, ctypes.byref(q), None) == minw.MINW_OK   # empty
    assert lib.aqe_forward(None, fake, 8, 0.5, ctypes.byref(q), None) == minw.MINW_EINVAL
    assert lib.aqe_forward(fake, fake, 8, 1.5, ctypes.byref(q), None) == minw.MINW_EINVAL
    bad = minw.quant(4)
    assert lib.aqe_forward(fake, fake, 8, 0.5, ctypes.byref(bad), None) == minw.MINW_EINVAL
    unordered = minw.quant(3, (0.1, 0.5, 0.2))
    assert lib.aqe_forward(fake, fake, 8, 0.5, ctypes.byref(unordered), None) == minw.MINW_EINVAL
    assert lib.aqe_backward(fake, fake, fake, -3, 0.5, None) == minw.MINW_EINVAL
    # misaligned pointer
    assert lib.aqe_backward(P(4100), fake, fake, 8, 0.5, None) == minw.MINW_EINVAL
    # convolution: C not a multiple of 32 is unsupported, bad bits invalid
    assert lib.minw_conv2d(fake, 1, 48, 8, 8, 1, fake, 4, 3, 3, 1, 1, 1, fake, None, None, None, 0,
                           None) == minw.MINW_EUNSUPPORTED
    assert lib.minw_conv2d(fake, 1, 64, 8, 8, 4, fake, 4, 3, 3, 1, 1, 1, fake, None, None, None, 0,
                           None) == minw.MINW_EINVAL
    assert lib.minw_conv2d(fake, 1, 64, 8, 8, 1, fake, 4, 3, 3, 1, 1, 1, None, None, None, None, 0,
                           None) == minw.MINW_EINVAL
    # y_out without its BN parameters
    assert lib.minw_conv2d(fake, 1, 64, 8, 8, 1, fake, 4, 3, 3, 1, 1, 1, None, None, None, fake, 0,
                           None) == minw.MINW_EINVAL
    # odd pooled size
    qo = minw.quant(1)
    assert lib.minw_conv_block(fake, 1, 64, 7, 7, 1, fake, 4, 3, 3, 1, 1, 1, 1, fake, fake,
                               ctypes.byref(qo), fake, None, 0, None) == minw.MINW_EUNSUPPORTED
    # network: too few layers / null output handle
    assert lib.minw_net_create(None, 0, 1, 0, None, None) == minw.MINW_EINVAL


def test_pointer_marshalling_rejects_host_tensors():
    torch = pytest.importorskip("torch")
    from paper_2003_04296_gb300 import minw
    with pytest.raises(ValueError):
        minw._ptr(torch.zeros(4))


def _al256(x):
    return (x + 255) // 256 * 256


def test_train_workspace_layout(lib):
    """minw_fc_train_workspace_bytes is the documented regions, each 256-byte
    aligned (bf16 W^, W^T padded to Op = O rounded up to 64, a, a^T, fp32 a~,
    bf16 g~ and g~^T, the two unit BN vectors), plus the K-slice partial sums
    of the products that split: none for a short reduction, whole slices of
    the forward product's 128 x 256-column tiles otherwise.  Invalid sizes
    give 0, and the step rejects sizes it does not support on the host."""
    from paper_2003_04296_gb300 import minw

    def regions(B, K, O):
        Op = (O + 63) // 64 * 64
        M = max(K, O)
        parts = [2 * O * K, 2 * K * Op, 2 * B * K, 2 * K * B, 4 * B * O, 2 * B * Op, 2 * O * B, 4 * M, 4 * M]
        return sum(_al256(p) for p in parts)

    for B, K, O in [(64, 128, 96), (128, 256, 10), (256, 512, 512)]:      # reductions under 16 K blocks: no split
        assert minw.minw_fc_train_workspace_bytes(B, K, O) == regions(B, K, O)
    for B, K, O in [(256, 1024, 512), (256, 8192, 1024)]:
        # the split region: the forward product's breakpoint area (O x 7 floats) and
        # whole slices of its 128 x 256-column tiles, 3 .. nk / 4 of them
        extra = minw.minw_fc_train_workspace_bytes(B, K, O) - regions(B, K, O)
        tiles = ((B + 127) // 128) * ((O + 255) // 256)
        slice_bytes = tiles * 128 * 256 * 4
        ks, rem = divmod(extra - _al256(28 * O), slice_bytes)
        assert rem == 0 and 3 <= ks <= (K // 64) // 4, (B, K, O, ks, rem)
    for bad in [(0, 128, 8), (64, 0, 8), (64, 128, 0), (-1, 128, 8)]:
        assert minw.minw_fc_train_workspace_bytes(*bad) == 0
    P = ctypes.c_void_p
    fake = P(4096)
    q = minw.quant(1)
    args = lambda B_, K_, O_, alpha=0.5: (fake, fake, fake, B_, K_, O_, alpha, 0.1, ctypes.byref(q), None, fake,
                                          None, None, fake, 1 << 30, None)
    assert lib.minw_fc_train_step(*args(64, 100, 8)) == minw.MINW_EUNSUPPORTED     # K % 64
    assert lib.minw_fc_train_step(*args(48, 128, 8)) == minw.MINW_EUNSUPPORTED     # B % 64
    assert lib.minw_fc_train_step(*args(64, 128, 8, alpha=1.5)) == minw.MINW_EINVAL
    assert lib.minw_fc_train_step(P(4100), fake, fake, 64, 128, 8, 0.5, 0.1, ctypes.byref(q), None, fake, None,
                                  None, fake, 1 << 30, None) == minw.MINW_EINVAL   # misaligned A
    assert lib.minw_fc_train_step(fake, fake, fake, 64, 128, 8, 0.5, 0.1, ctypes.byref(q), None, fake, None,
                                  None, fake, 16, None) == minw.MINW_EINVAL        # workspace too small
