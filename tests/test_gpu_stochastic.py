"""GPU parity of the stochastic AQE forward (Eq. our: alpha sign(a - z) +
(1 - alpha) a, z ~ U[-1, 1) from Philox4x64-10) against the oracle through the
C ABI: every element's decision equals the oracle's (its noise is a pure
function of seed, offset and index), the values within the fp32 tolerance, at
ragged sizes, several seeds and offsets, and the full 256 x 512 x 14 x 14
tensor of the bit-width sweep; then Theorem 1's expectation on the GPU's own
draws, and the argument checks."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import aqe_problem  # noqa: E402
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


def _check(x_np, y_gpu, alpha, seed, offset):
    ref, z = O.aqe_forward_stochastic(x_np, alpha, seed, offset)
    got = y_gpu.cpu().numpy()
    # a flipped decision moves the value by 2 alpha, far outside the tolerance
    assert_close(got, ref)
    if alpha > 0:
        s = np.where(got - (1.0 - alpha) * x_np.astype(np.float64) > 0, 1.0, -1.0)
        assert np.array_equal(s > 0, x_np.astype(np.float64) > z)


@pytest.mark.parametrize("n", [1, 7, 8, 9, 4097, (1 << 20) + 5])
@pytest.mark.parametrize("alpha,seed,offset", [(0.75, 1, 0), (0.5, 2**63 + 5, 2**64 - 3), (1.0, 77, 1000)])
def test_stochastic_forward(dev, M, n, alpha, seed, offset):
    p = aqe_problem(300 + n, n)
    x = dev_tensor(p["x"], dev)
    y = torch.empty_like(x)
    M.aqe_forward_stochastic(x, y, alpha, seed, offset)
    torch.cuda.synchronize()
    _check(p["x"], y, alpha, seed, offset)


def test_stochastic_forward_full_sweep_tensor(dev, M):
    """The 256 x 512 x 14 x 14 tensor of the bit-width sweep (25.7 M elements),
    every element against the oracle; two calls with offsets ceil(n / 8) apart
    draw the noise of disjoint counter blocks."""
    n = 256 * 512 * 14 * 14
    p = aqe_problem(55, n)
    x = dev_tensor(p["x"], dev)
    y = torch.empty_like(x)
    for k in range(2):
        off = 11 + k * ((n + 7) // 8)
        M.aqe_forward_stochastic(x, y, 0.75, 2026, off)
        torch.cuda.synchronize()
        _check(p["x"], y, 0.75, 2026, off)


def test_stochastic_theorem1_on_gpu(dev, M):
    """E_z[sign(a - z)] = max(-1, min(1, a)) on the GPU's draws (Monte Carlo,
    2^22 draws per value, within 5 sigma)."""
    m = 1 << 22
    for j, a in enumerate([-1.25, -0.4, 0.0, 0.6, 1.5]):
        x = torch.full((m,), a, dtype=torch.float32, device=dev)
        y = torch.empty_like(x)
        M.aqe_forward_stochastic(x, y, 0.5, 500 + j, 0)
        s = ((y.double() - 0.5 * float(np.float32(a))) / 0.5).cpu().numpy()
        np.testing.assert_allclose(np.abs(s), 1.0, rtol=0, atol=1e-6)
        exact = float(np.clip(np.float32(a), -1.0, 1.0))
        sig = np.sqrt(max(1 - exact ** 2, 1e-12) / m)
        assert abs(s.mean() - exact) <= 5 * sig + 2.0 ** -22


def test_stochastic_forward_errors(dev, M):
    x = torch.zeros(64, dtype=torch.float32, device=dev)
    y = torch.empty_like(x)
    with pytest.raises(M.MinwError):
        M.aqe_forward_stochastic(x, y, 1.5, 0, 0)
    with pytest.raises(M.MinwError):
        M.aqe_forward_stochastic(x[1:], y[1:], 0.5, 0, 0)          # 4-byte offset: not 16-byte aligned
