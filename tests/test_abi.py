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
