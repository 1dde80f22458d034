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


def test_weight_only_nets_host_validation(lib):
    """minw_wdense_create, minw_wresnet_create, minw_wdense_features and
    minw_conv2d_bf16_hardtanh reject bad arguments before any device call."""
    from paper_2003_04296_gb300 import minw
    P = ctypes.c_void_p
    fake = 4096                        # never dereferenced: validation fails first
    out = P()

    def dense(**kw):
        d = minw.WDenseDesc()
        d.layers, d.growth, d.bits_w, d.image_hw, d.num_classes = 16, 12, 3, 32, 10
        for i, t in enumerate((0.75, 0.375, 0.125)):
            d.thr_w[i] = t
        d.stem_w = d.stem_scale = d.stem_shift = d.fc_w = d.fc_scale = d.fc_shift = fake
        for j in range(3 * minw.WDENSE_MAX_LAYERS):
            d.b_w[j] = d.b_scale[j] = d.b_shift[j] = d.c_w[j] = d.c_scale[j] = d.c_shift[j] = fake
        for i in range(2):
            d.t_w[i] = d.t_scale[i] = d.t_shift[i] = fake
        for k, v in kw.items():
            setattr(d, k, v)
        return d

    create = lambda d, mb=8: lib.minw_wdense_create(ctypes.byref(d), mb, None, ctypes.byref(out))
    assert create(dense(), 0) == minw.MINW_EINVAL                       # batch
    for bad in (dict(layers=0), dict(layers=minw.WDENSE_MAX_LAYERS + 1), dict(growth=0), dict(growth=65),
                dict(bits_w=4), dict(image_hw=30), dict(image_hw=4), dict(num_classes=0), dict(stem_w=None)):
        assert create(dense(**bad)) == minw.MINW_EINVAL, bad
    d = dense()
    d.c_shift[3 * 16 - 1] = None                                        # last layer's BN shift missing
    assert create(d) == minw.MINW_EINVAL
    d = dense()
    d.thr_w[0], d.thr_w[2] = 0.1, 0.5                                   # thresholds not descending
    assert create(d) == minw.MINW_EINVAL
    # 32 layers of growth 64 end on 3616 channels: more than the head stages
    assert create(dense(layers=32, growth=64)) == minw.MINW_EUNSUPPORTED
    assert lib.minw_wdense_create(None, 8, None, ctypes.byref(out)) == minw.MINW_EINVAL
    r = minw.WResNetDesc()
    r.n, r.bits_w, r.image_hw, r.num_classes = 0, 3, 32, 10
    assert lib.minw_wresnet_create(ctypes.byref(r), 8, None, ctypes.byref(out)) == minw.MINW_EINVAL
    c, row = ctypes.c_int32(), ctypes.c_int32()
    assert lib.minw_wdense_features(None, 0, P(fake), 1, ctypes.byref(c), ctypes.byref(row),
                                    None) == minw.MINW_EINVAL
    # the fused epilogue: a row too short for its channels, input rows shorter than C
    assert lib.minw_conv2d_bf16_hardtanh(P(fake), 1, 64, 4, 4, 0, P(fake), 8, 1, 1, 1, 1, 0, P(fake), P(fake),
                                         P(fake), 16, 10, None, None, None) == minw.MINW_EINVAL
    assert lib.minw_conv2d_bf16_hardtanh(P(fake), 1, 64, 4, 4, 32, P(fake), 8, 1, 1, 1, 1, 0, P(fake), P(fake),
                                         P(fake), 16, 0, None, None, None) == minw.MINW_EINVAL
    assert lib.minw_conv2d_bf16_hardtanh(P(fake), 1, 64, 4, 4, 0, P(fake), 8, 1, 1, 1, 1, 0, None, P(fake),
                                         P(fake), 16, 0, None, None, None) == minw.MINW_EINVAL
