"""GPU parity of Algorithm 1's training step on a fully connected layer,
through the C ABI.

The building blocks are checked stage by stage against the oracle fed with
the GPU's own inputs to each stage: the weight AQE forward and the activation
AQE, the backward masks and the update bit for bit (one fp32 operation each),
the bf16 conversions bit for bit, and the tensor-core products of given bf16
operands within the bound of fp32 accumulation, K 2^-23 (|P| |Q|) for a
product P Q with K terms.

minw_fc_train_step is then checked against the oracle's step at the paper's
precision (fp32 operands, fp64 sums).  The GPU forms its three products from
bf16 roundings of the fp32 operands, so each product P Q differs from the
exact one by at most

    (2^-7 + 2^-16 + K 2^-23 (1 + 2^-8)^2) (|P| |Q|) + 2^-24 |P Q|

(two operand roundings of relative size 2^-8 each, the fp32 accumulation, and
the oracle's own rounding to fp32).  The stages after the forward product are
compared with the oracle fed the GPU's forward product (its a_pre argument):
a_out bit for bit, g_in within the bound, the updated weights within lr 2 alpha
times the weight gradient's bound plus one fp32 ulp."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as O  # noqa: E402
from paper_2003_04296_gb300.inputs import DEFAULT_THR  # noqa: E402
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


def _bf16(t):
    u = t.cpu().numpy().view(np.uint16).astype(np.uint32) << 16
    return u.view(np.float32)


def _check_product(got, P, Q):
    """got ~ P @ Q (fp64 reference), within K 2^-23 (|P| @ |Q|)."""
    ref = P.astype(np.float64) @ Q.astype(np.float64)
    bound = P.shape[1] * 2.0 ** -23 * (np.abs(P).astype(np.float64) @ np.abs(Q).astype(np.float64)) + 1e-30
    err = np.abs(got.astype(np.float64) - ref)
    assert (err <= bound).all(), f"worst err/bound {np.max(err / bound)}"


def _problem(seed, B, K, O_):
    r = np.random.default_rng(seed)
    A = np.clip(r.standard_normal((B, K)), -1.5, 1.5).astype(np.float32)
    W = r.uniform(-1, 1, (O_, K)).astype(np.float32)
    G = (r.standard_normal((B, O_)) * 0.1).astype(np.float32)
    return A, W, G


CASES = [(64, 128, 96, 0.75, 1, 1), (128, 256, 10, 0.3, 3, 2), (256, 1024, 512, 0.6, 2, 1)]


@pytest.mark.parametrize("case", CASES)
def test_train_stages(dev, M, case):
    B, K, O_, alpha, bw, ba = case
    A, W, G = _problem(sum(case[:3]), B, K, O_)
    Op = (O_ + 63) // 64 * 64
    qw, qa = M.quant(bw, DEFAULT_THR[bw]), M.quant(ba, DEFAULT_THR[ba])
    At, Wt, Gt = dev_tensor(A, dev), dev_tensor(W, dev), dev_tensor(G, dev)
    i16 = dict(dtype=torch.int16, device=dev)
    # forward: W^ (Eq. weight), the bf16 operands, a~, a_out (Eq. activation)
    what = torch.empty_like(Wt)
    M.aqe_forward(Wt, what, alpha, qw)
    what_np = what.cpu().numpy()
    assert np.array_equal(what_np, O.aqe_forward_f32(W, alpha, bw, DEFAULT_THR[bw]))
    wb, wtb = torch.empty((O_, K), **i16), torch.empty((K, Op), **i16)
    ab, atb = torch.empty((B, K), **i16), torch.empty((K, B), **i16)
    M.minw_bf16_matrix(what, wb)
    M.minw_bf16_matrix(what, wtb, transpose=True)
    M.minw_bf16_matrix(At, ab)
    M.minw_bf16_matrix(At, atb, transpose=True)
    Wq, Aq = O.bf16_round(what_np), O.bf16_round(A)
    assert np.array_equal(_bf16(wb), Wq) and np.array_equal(_bf16(ab), Aq)
    assert np.array_equal(_bf16(wtb)[:, :O_], Wq.T) and not _bf16(wtb)[:, O_:].any()
    assert np.array_equal(_bf16(atb), Aq.T)
    ones, zeros = torch.ones(max(K, O_), device=dev), torch.zeros(max(K, O_), device=dev)
    at = torch.empty((B, O_), dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(ab, B, K, 1, 1, wb, O_, 1, 1, bw, 1, 0, 0, ones, zeros, at)
    at_np = at.cpu().numpy()
    _check_product(at_np, Aq, Wq.T)
    a_out = torch.empty_like(at)
    M.aqe_forward(at, a_out, alpha, qa)
    assert np.array_equal(a_out.cpu().numpy(), O.aqe_forward_f32(at_np, alpha, ba, DEFAULT_THR[ba]))
    # backward: the mask of Eq. activation, g_in = g~ W^, g_W^ = g~^T A, Eq. weight's mask, the update
    gat = torch.empty_like(at)
    M.aqe_backward(at, Gt, gat, alpha)
    gat_np = gat.cpu().numpy()
    assert np.array_equal(gat_np, O.aqe_backward_f32(at_np, G, alpha))
    gb, gtb = torch.empty((B, Op), **i16), torch.empty((O_, B), **i16)
    M.minw_bf16_matrix(gat, gb)
    M.minw_bf16_matrix(gat, gtb, transpose=True)
    Gq = O.bf16_round(gat_np)
    assert np.array_equal(_bf16(gb)[:, :O_], Gq) and np.array_equal(_bf16(gtb), Gq.T)
    g_in = torch.empty((B, K), dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(gb, B, Op, 1, 1, wtb, K, 1, 1, bw, 1, 0, 0, ones, zeros, g_in)
    _check_product(g_in.cpu().numpy(), Gq, Wq)
    gwhat = torch.empty((O_, K), dtype=torch.float32, device=dev)
    M.minw_conv2d_bf16(gtb, O_, B, 1, 1, atb, K, 1, 1, bw, 1, 0, 0, ones, zeros, gwhat)
    gwhat_np = gwhat.cpu().numpy()
    _check_product(gwhat_np, Gq.T, Aq)
    gw = torch.empty_like(Wt)
    M.aqe_backward(Wt, gwhat, gw, alpha)
    gw_np = gw.cpu().numpy()
    assert np.array_equal(gw_np, O.aqe_backward_f32(W, gwhat_np, alpha))
    Wn = Wt.clone()
    M.minw_sgd_clip(Wn, gw, 0.05)
    assert np.array_equal(Wn.cpu().numpy(), O.sgd_clip(W, gw_np, 0.05))


def _step_bound(P, Q):
    """Bound of a bf16-operand tensor-core product against the exact product
    of the fp32 operands P [m][K] and Q [K][n] (the module docstring)."""
    P64, Q64 = P.astype(np.float64), Q.astype(np.float64)
    K = P.shape[1]
    mag = np.abs(P64) @ np.abs(Q64)
    return (2.0 ** -7 + 2.0 ** -16 + K * 2.0 ** -23 * (1 + 2.0 ** -8) ** 2) * mag + 2.0 ** -24 * np.abs(P64 @ Q64) + 1e-30


def _within(got, ref, bound, what):
    err = np.abs(got.astype(np.float64) - ref.astype(np.float64))
    assert (err <= bound).all(), f"{what}: worst err/bound {np.max(err / bound)}"


@pytest.mark.parametrize("case", CASES + [(256, 8192, 1024, 0.75, 1, 1), (1152, 256, 256, 0.5, 1, 2)])
@pytest.mark.parametrize("last", [False, True])
def test_train_step(dev, M, case, last):
    """minw_fc_train_step against the oracle's Algorithm 1 step at the paper's
    precision.  a~ (a_pre, or a_out for the last layer) lies within the
    bf16-operand bound of the oracle's a~; with the GPU's a~ substituted, a_out
    equals the oracle's bit for bit, g_in lies within the bound of g~ W^, and
    the updated W within lr 2 alpha times the bound of g~^T A plus one fp32 ulp.
    (256, 8192, 1024) is fc1 of the CIFAR model at the training bench's batch,
    whose forward product splits along K; at (1152, 256, 256) the weight
    gradient's product (contraction over the batch: 18 K blocks, 256 output
    rows) runs on CTA pairs with the update in their staged-store epilogue.  A second step from the same inputs
    gives the same bits (the K slices add in a fixed order)."""
    B, K, O_, alpha, bw, ba = case
    lr = 0.05
    A, W, G = _problem(7 + sum(case[:3]), B, K, O_)
    qw, qa = M.quant(bw, DEFAULT_THR[bw]), (None if last else M.quant(ba, DEFAULT_THR[ba]))
    q_a = None if last else (ba, DEFAULT_THR[ba])
    At, Gt = dev_tensor(A, dev), dev_tensor(G, dev)
    ws = torch.empty(M.minw_fc_train_workspace_bytes(B, K, O_), dtype=torch.uint8, device=dev)
    outs = []
    for _ in range(2):
        W1 = dev_tensor(W, dev)
        a1, g1, pre = (torch.empty((B, O_), device=dev), torch.empty((B, K), device=dev),
                       torch.empty((B, O_), device=dev))
        M.minw_fc_train_step(At, W1, Gt, alpha, lr, qw, qa, a1, g1, ws, a_pre=pre)
        torch.cuda.synchronize()
        outs.append((W1.cpu().numpy(), a1.cpu().numpy(), g1.cpu().numpy(), pre.cpu().numpy()))
    W1, a1, g1, pre = outs[0]
    for x, y in zip(outs[0], outs[1][:3]):
        assert np.array_equal(x, y)
    at = a1 if last else pre
    # the forward product against the paper-precision oracle's
    what = O.aqe_forward_f32(W, alpha, bw, DEFAULT_THR[bw])
    ref = O.fc_train_step(A, W, G, alpha, lr, bw, DEFAULT_THR[bw], q_a)
    _within(at, ref[3], _step_bound(A, what.T), "a~")
    # the later stages with the GPU's a~ substituted
    a_ref, gin_ref, W_ref, _ = O.fc_train_step(A, W, G, alpha, lr, bw, DEFAULT_THR[bw], q_a, a_pre=at)
    if not last:
        assert np.array_equal(a1, a_ref)
    gat = G if last else O.aqe_backward_f32(at, G, alpha)
    _within(g1, gin_ref, _step_bound(gat, what), "g_in")
    gb = _step_bound(gat.T, A)
    gw_ref = gat.T.astype(np.float64) @ A.astype(np.float64)
    _within(W1, W_ref, lr * 2 * alpha * (gb + 2.0 ** -24 * np.abs(gw_ref)) + 2.0 ** -23, "W")
    assert np.abs(W1).max() <= 1.0


def test_train_step_errors(dev, M):
    A = torch.zeros((64, 100), device=dev)
    W = torch.zeros((8, 100), device=dev)
    G = torch.zeros((64, 8), device=dev)
    ws = torch.empty(1 << 20, dtype=torch.uint8, device=dev)
    with pytest.raises(M.MinwError):       # K % 64 != 0
        M.minw_fc_train_step(A, W, G, 0.5, 0.1, M.quant(1), None, torch.empty((64, 8), device=dev), None, ws)
