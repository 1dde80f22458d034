"""numpy front-end of the C oracle (test infrastructure only).

Only tests/, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` leg of
``bench.py`` may import this module.  Each function hands plain numpy arrays
to the single-threaded C routines of ``minw_oracle.c`` and returns numpy
arrays; nothing here touches a GPU or the CUDA library.

Conventions
-----------
* Activations are NCHW fp32, weights OIHW fp32 (latent, full precision).
* ``thr`` holds the quantizer thresholds D_1 > D_2 > D_3 (unused entries 0).
* Levels come back dequantized (fp64): {-1, 1}, {-1, 0, 1} or
  {0, +-1/4, +-1/2, +-1} for 1, 2 and 3 bits (Sec. IV-A).
* An integer accumulator ``acc`` is the real dot product times
  2^(f_a + f_w) with f = 2 for a 3-bit operand and 0 otherwise.
"""
import ctypes
import numpy as np

from . import build as _build

_lib = None


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        P = ctypes.c_void_p
        i32, i64, f32, f64 = ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_double
        L.orc_h.restype = f64
        L.orc_h.argtypes = [f32, i32, P, f32]
        L.orc_qnn.restype = f64
        L.orc_qnn.argtypes = [f64, i32, P]
        L.orc_quantize.argtypes = [P, i64, i64, i32, P, P, P]
        L.orc_aqe_forward.argtypes = [P, i64, f64, i32, P, f32, P]
        L.orc_aqe_backward.argtypes = [P, P, i64, f64, P]
        L.orc_aqe_forward_f32.argtypes = [P, i64, f32, i32, P, f32, P]
        L.orc_aqe_backward_f32.argtypes = [P, P, i64, f32, P]
        L.orc_sgd_clip.argtypes = [P, P, i64, f32]
        u64 = ctypes.c_uint64
        L.orc_philox4x64_10.argtypes = [P, P, P]
        L.orc_aqe_forward_stochastic.argtypes = [P, i64, f64, u64, u64, P, P]
        L.orc_pack.argtypes = [P, i32, i32, i32, i32, i32, P]
        L.orc_bf16_round.restype = f32
        L.orc_bf16_round.argtypes = [f32]
        L.orc_bf16_round_array.argtypes = [P, i64, P]
        L.orc_conv2d_real.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, i32, i32, P]
        L.orc_conv2d_input_grad.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, i32, i32, i32, i32, P]
        L.orc_conv2d_weight_grad.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, i32, i32, i32, i32, P]
        L.orc_conv2d.restype = i32
        L.orc_conv2d.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, i32, i32, i32, P]
        L.orc_maxpool_i32.argtypes = [P, i32, i32, i32, i32, i32, i32, P]
        L.orc_maxpool_f32.argtypes = [P, i32, i32, i32, i32, i32, i32, i32, P]
        L.orc_affine_i32.argtypes = [P, i32, i32, i32, P, P, P]
        L.orc_affine_f32.argtypes = [P, i32, i32, i32, P, P, P]
        L.orc_hardtanh.argtypes = [P, i64]
        L.orc_conv2d_f32_seq.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, i32, i32, P]
        L.orc_avgpool_f32.argtypes = [P, i32, i32, i32, P]
        L.orc_linear_f32_seq.argtypes = [P, i32, i32, P, i32, P, P]
        _lib = L
    return _lib


def _p(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _thr(thr):
    t = np.zeros(3, dtype=np.float32)
    if thr is not None:
        v = np.asarray(thr, dtype=np.float32).ravel()
        t[: v.size] = v
    return t


def units_shift(bits):
    """f in acc = real * 2^(f_a + f_w): 3-bit levels are multiples of 1/4."""
    return 2 if bits == 3 else 0


def h(x, bits, thr=None, scale=1.0):
    """Level function h of Eq. sign / Eq. tnn / Eq. qnn on a scalar fp32 input."""
    t = _thr(thr)
    return lib().orc_h(float(np.float32(x)), bits, _p(t), float(np.float32(scale)))


def qnn(u, n, thr):
    """Eq. qnn for an n-bit QNN with q = 2^(n-1)-1 thresholds (fp64 input)."""
    t = np.ascontiguousarray(np.asarray(thr, dtype=np.float64).ravel())
    if t.size == 0:
        t = np.zeros(1)
    return lib().orc_qnn(float(u), int(n), _p(t))


def quantize(x, bits, thr=None, scale=None):
    """Eq. inference: dequantized levels h(x * scale) with one scale per
    leading index (``scale`` of length x.shape[0]) or scale 1."""
    x = _f32(x)
    out = np.empty(x.shape, dtype=np.float64)
    t = _thr(thr)
    n_outer = x.shape[0] if scale is not None else 1
    n_inner = x.size // max(n_outer, 1)
    s = _f32(scale) if scale is not None else None
    lib().orc_quantize(_p(x), n_outer, n_inner, bits, _p(t),
                       _p(s) if s is not None else None, _p(out))
    return out


def aqe_forward(x, alpha, bits, thr=None, scale=1.0):
    """Eq. ours / Eq. activation forward in fp64."""
    x = _f32(x)
    y = np.empty(x.shape, dtype=np.float64)
    t = _thr(thr)
    lib().orc_aqe_forward(_p(x), x.size, float(alpha), bits, _p(t),
                          float(np.float32(scale)), _p(y))
    return y


def aqe_backward(x, g, alpha):
    """Eq. activation / Eq. weight backward in fp64."""
    x = _f32(x)
    g = _f32(g)
    gx = np.empty(x.shape, dtype=np.float64)
    lib().orc_aqe_backward(_p(x), _p(g), x.size, float(alpha), _p(gx))
    return gx


def aqe_forward_f32(x, alpha, bits, thr=None, scale=1.0):
    """Eq. activation / Eq. weight forward in the fp32 operations of a training
    step: fmaf(alpha, h(x), (1 - alpha) x), each product rounded to fp32."""
    x = _f32(x)
    y = np.empty(x.shape, dtype=np.float32)
    lib().orc_aqe_forward_f32(_p(x), x.size, float(np.float32(alpha)), bits, _p(_thr(thr)),
                              float(np.float32(scale)), _p(y))
    return y


def aqe_backward_f32(x, g, alpha):
    """Eq. activation / Eq. weight backward in fp32: (|x| <= 1) ? g (2 alpha) : 0."""
    x, g = _f32(x), _f32(g)
    gx = np.empty(x.shape, dtype=np.float32)
    lib().orc_aqe_backward_f32(_p(x), _p(g), x.size, float(np.float32(alpha)), _p(gx))
    return gx


def sgd_clip(w, g, lr):
    """Algorithm 1's update with a plain gradient step: min(1, max(-1, w - lr g))
    (one fmaf), returned as a new fp32 array."""
    w = _f32(w).copy()
    g = _f32(g)
    lib().orc_sgd_clip(_p(w), _p(g), w.size, float(np.float32(lr)))
    return w


def philox4x64_10(counter, key):
    """Philox4x64-10 block (Salmon et al., SC 2011): 4 x uint64 counter,
    2 x uint64 key -> 4 x uint64."""
    c = np.ascontiguousarray(counter, dtype=np.uint64)
    k = np.ascontiguousarray(key, dtype=np.uint64)
    out = np.empty(4, dtype=np.uint64)
    lib().orc_philox4x64_10(_p(c), _p(k), _p(out))
    return out


def aqe_forward_stochastic(x, alpha, seed, offset=0):
    """Eq. our: alpha sign(a - z) + (1 - alpha) a in fp64, z ~ U[-1, 1) drawn
    from Philox4x64-10 (element i: counter offset + i // 8, key (seed, 0),
    32-bit word i mod 8).  Returns (y, z)."""
    x = _f32(x)
    y = np.empty(x.shape, dtype=np.float64)
    z = np.empty(x.shape, dtype=np.float32)
    lib().orc_aqe_forward_stochastic(_p(x), x.size, float(alpha), int(seed) & (2**64 - 1),
                                     int(offset) & (2**64 - 1), _p(y), _p(z))
    return y, z


def pack(levels, bits):
    """Bit-plane packing of NCHW (or OIHW) dequantized levels into
    uint32 [N][H][W][bits][ceil(C/32)]."""
    lv = np.ascontiguousarray(levels, dtype=np.float64)
    N, C, H, W = lv.shape
    nw = (C + 31) // 32
    out = np.empty((N, H, W, bits, nw), dtype=np.uint32)
    lib().orc_pack(_p(lv), N, C, H, W, bits, _p(out))
    return out


def conv2d_levels(a_lv, w_lv, stride, pad, bits_a, bits_w):
    """Algorithm 1 inference product a~ = a^q W^q as a zero-padded fp64
    convolution of dequantized levels, returned as integer accumulators."""
    a = np.ascontiguousarray(a_lv, dtype=np.float64)
    w = np.ascontiguousarray(w_lv, dtype=np.float64)
    B, C, H, W = a.shape
    O, Cw, kh, kw = w.shape
    assert C == Cw
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (W + 2 * pad - kw) // stride + 1
    acc = np.empty((B, O, Ho, Wo), dtype=np.int32)
    rc = lib().orc_conv2d(_p(a), B, C, H, W, _p(w), O, kh, kw, stride, pad,
                          units_shift(bits_a) + units_shift(bits_w), _p(acc))
    if rc != 0:
        raise ArithmeticError("non-integral accumulator")
    return acc


def bf16_round(x):
    """fp32 -> bf16 (round to nearest, ties to even), returned as fp32 values."""
    x = _f32(x)
    out = np.empty(x.shape, dtype=np.float32)
    lib().orc_bf16_round_array(_p(x), x.size, _p(out))
    return out


def bf16_round_scalar(v):
    """bf16_round of one value, through the scalar C routine."""
    return float(lib().orc_bf16_round(float(v)))


def fc_train_step(A, W, G, alpha, lr, bits_w, thr_w, q_a=None, a_pre=None):
    """One step of Algorithm 1 on a fully connected layer with input A [B][K],
    latent weights W [O][K] and upstream gradient G [B][O], in the order of
    Algorithm 1 and at its precision (Sec. III-C: the weights and activations
    entering the loss are full precision): the weight AQE W^ (Eq. weight,
    fp32), the forward product a~ = A W^T (fp64 sums of the fp32 operands,
    rounded to fp32), the activation AQE and its backward mask g~ (Eq.
    activation; skipped for the last layer, q_a None), the input gradient
    g_in = g~ W^ and the weight gradient g_W^ = g~^T A (fp64 sums of the fp32
    operands, rounded to fp32), then the mask of Eq. weight and the clipped
    update.  q_a = (bits, thr).

    a_pre, when given, replaces the forward product a~ for the rest of the
    step (a stage-wise check: the later stages of the oracle applied to the
    forward product another implementation computed).

    Returns (a_out, g_in, W_new, a_pre) as fp32 arrays."""
    A, W, G = _f32(A), _f32(W), _f32(G)
    what = aqe_forward_f32(W, alpha, bits_w, thr_w).astype(np.float64)
    A64 = A.astype(np.float64)
    if a_pre is None:
        a_pre = (A64 @ what.T).astype(np.float32)
    else:
        a_pre = _f32(a_pre)
    if q_a is None:
        a_out, g_t = a_pre, G
    else:
        a_out = aqe_forward_f32(a_pre, alpha, q_a[0], q_a[1])
        g_t = aqe_backward_f32(a_pre, G, alpha)
    g64 = g_t.astype(np.float64)
    g_in = (g64 @ what).astype(np.float32)
    g_w = (g64.T @ A64).astype(np.float32)
    W_new = sgd_clip(W, aqe_backward_f32(W, g_w, alpha), lr)
    return a_out, g_in, W_new, a_pre


def conv2d_real(a, w, stride, pad):
    """Zero-padded fp64 convolution of real activations a [B][C][H][W] with
    weights w [O][C][kh][kw] (the weight-only layers' exact accumulator)."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    w = np.ascontiguousarray(w, dtype=np.float64)
    B, C, H, W = a.shape
    O, Cw, kh, kw = w.shape
    assert C == Cw
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (W + 2 * pad - kw) // stride + 1
    out = np.empty((B, O, Ho, Wo), dtype=np.float64)
    lib().orc_conv2d_real(_p(a), B, C, H, W, _p(w), O, kh, kw, stride, pad, _p(out))
    return out


def conv2d_input_grad(g, w, stride, pad, H, W):
    """Algorithm 1's input gradient of a convolutional layer: the gradient of
    sum(g * conv2d_real(a, w)) with respect to a [B][C][H][W] (fp64)."""
    g = np.ascontiguousarray(g, dtype=np.float64)
    w = np.ascontiguousarray(w, dtype=np.float64)
    B, O, Ho, Wo = g.shape
    O2, C, kh, kw = w.shape
    assert O == O2
    ga = np.empty((B, C, H, W), dtype=np.float64)
    lib().orc_conv2d_input_grad(_p(g), B, O, Ho, Wo, _p(w), C, kh, kw, stride, pad, H, W, _p(ga))
    return ga


def conv2d_weight_grad(g, a, kh, kw, stride, pad):
    """Algorithm 1's weight gradient of a convolutional layer: the gradient of
    sum(g * conv2d_real(a, w)) with respect to w [O][C][kh][kw] (fp64)."""
    g = np.ascontiguousarray(g, dtype=np.float64)
    a = np.ascontiguousarray(a, dtype=np.float64)
    B, O, Ho, Wo = g.shape
    B2, C, H, W = a.shape
    assert B == B2
    gw = np.empty((O, C, kh, kw), dtype=np.float64)
    lib().orc_conv2d_weight_grad(_p(g), B, O, Ho, Wo, _p(a), C, H, W, kh, kw, stride, pad, _p(gw))
    return gw


def conv_train_step(A, W, G, alpha, lr, bits_w, thr_w, stride, pad, q_a=None, a_pre=None):
    """Algorithm 1 on a convolutional layer, in the order and at the precision
    of fc_train_step: the weight AQE (fp32), the forward convolution of the
    fp32 operands (fp64 sums rounded to fp32), the activation AQE and its mask
    (q_a = (bits, thr); None for a layer without an activation quantizer), the
    input and weight gradients of the fp32 operands (fp64 sums rounded to
    fp32), then the mask of Eq. weight and the clipped update.  A [B][C][H][W],
    W [O][C][kh][kw], G [B][O][Ho][Wo]; a_pre as in fc_train_step.  Returns
    (a_out, g_in, W_new, a_pre)."""
    A, W, G = _f32(A), _f32(W), _f32(G)
    what = aqe_forward_f32(W, alpha, bits_w, thr_w).astype(np.float64)
    A64 = A.astype(np.float64)
    if a_pre is None:
        a_pre = conv2d_real(A64, what, stride, pad).astype(np.float32)
    else:
        a_pre = _f32(a_pre)
    if q_a is None:
        a_out, g_t = a_pre, G
    else:
        a_out = aqe_forward_f32(a_pre, alpha, q_a[0], q_a[1])
        g_t = aqe_backward_f32(a_pre, G, alpha)
    g64 = g_t.astype(np.float64)
    H, Wd = A.shape[2], A.shape[3]
    g_in = conv2d_input_grad(g64, what, stride, pad, H, Wd).astype(np.float32)
    g_w = conv2d_weight_grad(g64, A64, W.shape[2], W.shape[3], stride, pad).astype(np.float32)
    W_new = sgd_clip(W, aqe_backward_f32(W, g_w, alpha), lr)
    return a_out, g_in, W_new, a_pre


def maxpool_f64(x, k=2, s=2):
    """k x k / s max pooling of fp64 [B][C][H][W] (no padding)."""
    B, C, H, W = x.shape
    Ho, Wo = (H - k) // s + 1, (W - k) // s + 1
    out = np.full((B, C, Ho, Wo), -np.inf)
    for dy in range(k):
        for dx in range(k):
            out = np.maximum(out, x[:, :, dy:dy + s * (Ho - 1) + 1:s, dx:dx + s * (Wo - 1) + 1:s])
    return out


def maxpool_i32(acc, k=2, s=2):
    acc = np.ascontiguousarray(acc, dtype=np.int32)
    B, C, H, W = acc.shape
    out = np.empty((B, C, (H - k) // s + 1, (W - k) // s + 1), dtype=np.int32)
    lib().orc_maxpool_i32(_p(acc), B, C, H, W, k, s, _p(out))
    return out


def maxpool_f32(x, k, s, p):
    x = _f32(x)
    B, C, H, W = x.shape
    out = np.empty((B, C, (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1), dtype=np.float32)
    lib().orc_maxpool_f32(_p(x), B, C, H, W, k, s, p, _p(out))
    return out


def affine(acc, scale, shift):
    """Inference BN as y = fmaf(acc, scale[c], shift[c]) over [B][C][...]."""
    scale, shift = _f32(scale), _f32(shift)
    B, C = acc.shape[:2]
    HW = int(np.prod(acc.shape[2:])) if acc.ndim > 2 else 1
    y = np.empty(acc.shape, dtype=np.float32)
    if acc.dtype == np.int32:
        a = np.ascontiguousarray(acc)
        lib().orc_affine_i32(_p(a), B, C, HW, _p(scale), _p(shift), _p(y))
    else:
        a = _f32(acc)
        lib().orc_affine_f32(_p(a), B, C, HW, _p(scale), _p(shift), _p(y))
    return y


def hardtanh(y):
    y = np.array(y, dtype=np.float32, copy=True)
    lib().orc_hardtanh(_p(y), y.size)
    return y


def conv2d_f32_seq(x, w, stride, pad):
    """fp32 convolution, one fmaf chain per output over (ci, ky, kx)."""
    x, w = _f32(x), _f32(w)
    B, C, H, W = x.shape
    O, Cw, kh, kw = w.shape
    assert C == Cw
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (W + 2 * pad - kw) // stride + 1
    out = np.empty((B, O, Ho, Wo), dtype=np.float32)
    lib().orc_conv2d_f32_seq(_p(x), B, C, H, W, _p(w), O, kh, kw, stride, pad, _p(out))
    return out


def avgpool_f32(x):
    x = _f32(x)
    B, C = x.shape[:2]
    HW = x.size // (B * C)
    out = np.empty((B, C), dtype=np.float32)
    lib().orc_avgpool_f32(_p(x), B, C, HW, _p(out))
    return out


def linear_f32_seq(x, w, bias=None):
    x, w = _f32(x), _f32(w)
    B, K = x.shape
    O = w.shape[0]
    y = np.empty((B, O), dtype=np.float32)
    b = _f32(bias) if bias is not None else None
    lib().orc_linear_f32_seq(_p(x), B, K, _p(w), O, _p(b) if b is not None else None, _p(y))
    return y
