"""Helpers of the GPU parity tests (device transfers and views only)."""
import numpy as np
import torch


def dev_tensor(a, device):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def words(t):
    return t.cpu().numpy().view(np.uint32)


def planes_view(t, N, H, W, P, C):
    return words(t).reshape(N, H, W, P, (C + 31) // 32)


def assert_close(got, ref, rtol=1e-5, atol=1e-6):
    """The floating-point tolerance of the parity bar: 1e-5 relative and
    1e-6 absolute, element by element."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    bad = np.abs(got - ref) > atol + rtol * np.abs(ref)
    assert not bad.any(), f"{bad.sum()} of {bad.size} outside tolerance; worst {np.max(np.abs(got - ref))}"


def case_seed(*parts):
    """A seed fixed by a test case's parameters (crc32 of their repr: unlike
    hash(), the same in every process)."""
    import zlib
    return zlib.crc32(repr(parts).encode()) % 1000
