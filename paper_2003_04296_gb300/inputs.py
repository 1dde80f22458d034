"""Seeded synthetic inputs shared by the oracle tests, the CUDA tests and the
bench.  This module draws random numbers and shapes them; it holds none of
the method's arithmetic (no quantizer, no convolution, no epilogue).

Every generator uses numpy's PCG64 (``default_rng(seed)``) and returns plain
fp32 numpy arrays, so the oracle and the CUDA path always receive byte-identical
data.  The tensors stand in for CIFAR-10/100 and ImageNet, which are not
available here: shapes and value ranges follow the paper's workloads
(Sec. IV: 3x32x32 CIFAR images, 224x224 ImageNet crops, Model A ConvNet,
ResNet-18), the distributions are synthetic.
"""
import numpy as np

# Default thresholds of the quantizers (the paper gives none): midpoints
# between adjacent levels, i.e. round to the nearest level, ties to the
# smaller magnitude.  2-bit: {-1, 0, 1}; 3-bit: {0, +-1/4, +-1/2, +-1}.
DEFAULT_THR = {1: (0.0, 0.0, 0.0), 2: (0.5, 0.0, 0.0), 3: (0.75, 0.375, 0.125)}

# Rough second moment of a level drawn from each quantizer on a unit-spread
# input; used only to give the synthetic BN statistics a plausible size.
_LEVEL_MS = {0: 1.0 / 3.0, 1: 1.0, 2: 0.5, 3: 0.25}


def rng(seed):
    return np.random.default_rng(seed)


def f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def weight_prescale(w, bits_w):
    """Per-output-channel multiplier applied before a weight quantizer with
    more than one non-zero magnitude: 1 / max|W[o]| maps each latent channel
    onto [-1, 1] (the range the paper clips latent weights to).  1-bit
    weights keep 1 (sign is scale invariant)."""
    O = w.shape[0]
    if bits_w == 1:
        return np.ones(O, dtype=np.float32)
    m = np.abs(w.reshape(O, -1).astype(np.float64)).max(axis=1)
    m[m == 0] = 1.0
    return f32(1.0 / m)


def bn_affine(r, O, fan_in, bits_in, bits_w, w_prescale, units_shift):
    """Synthetic inference-mode batch normalisation folded to a per-channel
    affine map on the layer's raw output: gamma ~ N(1, 0.1), beta ~ N(0, 0.1),
    running mean 0, running variance ~ fan_in times the level second moments.
    The returned scale also carries the accumulator unit 2^-units_shift and the
    weight prescale, so that y = scale * acc + shift."""
    gamma = r.normal(1.0, 0.1, O)
    beta = r.normal(0.0, 0.1, O)
    var = fan_in * _LEVEL_MS[bits_in] * _LEVEL_MS[bits_w]
    s = gamma / np.sqrt(var + 1e-5)
    s = s * (2.0 ** -units_shift) / w_prescale.astype(np.float64)
    return f32(s), f32(beta)


def _units(bits):
    return 2 if bits == 3 else 0


def conv_problem(seed, B, C, H, W, O, kh=3, kw=3, stride=1, pad=1, bits_a=1,
                 bits_w=1, x_dist="normal", w_sigma=0.05, bn=True):
    """One standalone quantized convolution: activations, latent weights,
    quantizer thresholds, weight prescale and the epilogue affine map."""
    r = rng(seed)
    if x_dist == "normal":
        x = r.standard_normal((B, C, H, W))
    elif x_dist == "absnormal_clip":          # |N(0,1)| clipped to [0, 1]
        x = np.minimum(np.abs(r.standard_normal((B, C, H, W))), 1.0)
    elif x_dist == "uniform":
        x = r.uniform(-1.0, 1.0, (B, C, H, W))
    else:
        raise ValueError(x_dist)
    w = r.normal(0.0, w_sigma, (O, C, kh, kw))
    x, w = f32(x), f32(w)
    ws = weight_prescale(w, bits_w)
    if bn:
        scale, shift = bn_affine(r, O, C * kh * kw, bits_a, bits_w, ws,
                                 _units(bits_a) + _units(bits_w))
    else:
        scale, shift = f32(np.ones(O)), f32(np.zeros(O))
    return dict(x=x, w=w, w_scale=ws, thr_a=DEFAULT_THR[bits_a],
                thr_w=DEFAULT_THR[bits_w], scale=scale, shift=shift,
                B=B, C=C, H=H, W=W, O=O, kh=kh, kw=kw, stride=stride, pad=pad,
                bits_a=bits_a, bits_w=bits_w)


def aqe_problem(seed, n, alpha=0.75):
    """AQE forward/backward operands: x ~ N(0, 1), upstream gradient g ~ N(0, 1)."""
    r = rng(seed)
    x = f32(r.standard_normal(n))
    g = f32(r.standard_normal(n))
    return dict(x=x, g=g, alpha=alpha)


def convnet_params(seed, bits_a=1, bits_w=1, widths=(128, 128, 256, 256, 512, 512),
                   pools=(False, True, False, True, False, True), fcs=(1024, 1024),
                   classes=10, in_ch=3, hw=32, w_sigma=0.05):
    """Model-A-shaped ConvNet (Sec. IV-B): six 3x3 convolutions with a 2x2 max
    pool after every second one, then three fully connected layers.  The first
    convolution sees the fp32 image, every weight is quantized, the last layer
    emits fp32 logits.  Each layer record holds latent fp32 weights and the
    folded BN affine map of its output."""
    r = rng(seed)
    layers = []
    c_in, size = in_ch, hw
    for i, (c_out, pool) in enumerate(zip(widths, pools)):
        bits_in = 0 if i == 0 else bits_a
        w = f32(r.normal(0.0, w_sigma, (c_out, c_in, 3, 3)))
        ws = weight_prescale(w, bits_w)
        u = (0 if bits_in == 0 else _units(bits_in)) + _units(bits_w)
        scale, shift = bn_affine(r, c_out, c_in * 9, bits_in, bits_w, ws, u)
        layers.append(dict(kind="conv", w=w, w_scale=ws, scale=scale, shift=shift,
                           pool=pool, bits_in=bits_in, bits_w=bits_w,
                           bits_out=bits_a, C=c_in, O=c_out, H=size, W=size,
                           kh=3, kw=3, stride=1, pad=1))
        c_in = c_out
        if pool:
            size //= 2
    k = c_in * size * size
    dims = list(fcs) + [classes]
    for j, o in enumerate(dims):
        w = f32(r.normal(0.0, w_sigma, (o, k)))
        ws = weight_prescale(w, bits_w)
        scale, shift = bn_affine(r, o, k, bits_a, bits_w, ws, _units(bits_a) + _units(bits_w))
        last = j == len(dims) - 1
        rec = dict(kind="fc", w=w, w_scale=ws, scale=scale, shift=shift, pool=False,
                   bits_in=bits_a, bits_w=bits_w, bits_out=0 if last else bits_a,
                   K=k, O=o)
        if j == 0:
            rec["in_shape"] = (c_in, size, size)   # flattened in (c, h, w) order
        layers.append(rec)
        k = o
    return dict(layers=layers, bits_a=bits_a, bits_w=bits_w,
                thr_a=DEFAULT_THR[bits_a], thr_w=DEFAULT_THR[bits_w],
                in_shape=(in_ch, hw, hw))


def convnet_input(seed, B, in_ch=3, hw=32):
    """CIFAR-shaped synthetic images, U(-1, 1)."""
    return f32(rng(seed).uniform(-1.0, 1.0, (B, in_ch, hw, hw)))
