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


# Expected maximum of k independent standard normals (k = 4: a 2x2 pool,
# k = 9: a 3x3 pool): the running mean a BN after a max pool would learn, in
# units of the pre-pool standard deviation.
POOL_MEAN = {1: 0.0, 4: 1.0294, 9: 1.4850}


def weight_ms(w, w_prescale, bits_w):
    """Per-output-channel second moment of the prescaled latent weights, a
    stand-in for the second moment of their levels (1 for sign weights)."""
    O = w.shape[0]
    if bits_w == 1:
        return np.ones(O)
    v = w.reshape(O, -1).astype(np.float64) * w_prescale.astype(np.float64)[:, None]
    return np.maximum((v * v).mean(axis=1), 1e-6)


def bn_affine(r, O, fan_in, bits_in, bits_w, w_prescale, units_shift, w_ms=None, pool_k=1):
    """Synthetic inference-mode batch normalisation folded to a per-channel
    affine map on the layer's raw output: gamma ~ N(1, 0.1), beta ~ N(0, 0.1),
    running variance ~ fan_in times the input and weight second moments
    (``w_ms`` per channel, else the level second moment of ``bits_w``),
    running mean 0, or the expected window maximum when a k-element max pool
    precedes the BN.  The returned scale also carries the accumulator unit
    2^-units_shift, so that y = scale * acc + shift.  Without ``w_ms`` the
    statistics are those of the latent-weight output (the scale also undoes
    the weight prescale); with it, those of the level output itself."""
    gamma = r.normal(1.0, 0.1, O)
    beta = r.normal(0.0, 0.1, O)
    wm = _LEVEL_MS[bits_w] if w_ms is None else w_ms
    var = fan_in * _LEVEL_MS[bits_in] * wm
    inv = gamma / np.sqrt(var + 1e-5)
    shift = beta - inv * POOL_MEAN[pool_k] * np.sqrt(var)
    s = inv * (2.0 ** -units_shift)
    if w_ms is None:
        s = s / w_prescale.astype(np.float64)
    return f32(s), f32(shift)


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


# The ConvNets of Sec. IV-B: Model A, then B with half the channels of every
# convolution, C with B's convolutions and half the units of the hidden fully
# connected layers, D with half of C's.
CIFAR_MODELS = {
    "A": dict(widths=(128, 128, 256, 256, 512, 512), fcs=(1024, 1024)),
    "B": dict(widths=(64, 64, 128, 128, 256, 256), fcs=(1024, 1024)),
    "C": dict(widths=(64, 64, 128, 128, 256, 256), fcs=(512, 512)),
    "D": dict(widths=(64, 64, 128, 128, 256, 256), fcs=(256, 256)),
}


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
        scale, shift = bn_affine(r, c_out, c_in * 9, bits_in, bits_w, ws, u,
                                 w_ms=weight_ms(w, ws, bits_w), pool_k=4 if pool else 1)
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
        scale, shift = bn_affine(r, o, k, bits_a, bits_w, ws, _units(bits_a) + _units(bits_w),
                                 w_ms=weight_ms(w, ws, bits_w))
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


def resnet18_params(seed, bits_a=3, bits_w=3, classes=1000, hw=224, w_sigma=0.02):
    """ResNet-18-shaped MINW-Net (Table V's network): fp32 7x7/2 stem (fp32
    weights), eight basic blocks (widths 64-128-256-512, stride 2 and a 1x1
    shortcut entering stages 2-4) with quantized weights, fp32 classifier.
    Latent weights ~ N(0, w_sigma); BN maps as ``bn_affine``."""
    r = rng(seed)
    out = dict(bits_a=bits_a, bits_w=bits_w, thr_a=DEFAULT_THR[bits_a], thr_w=DEFAULT_THR[bits_w],
               classes=classes, hw=hw)
    sw = f32(r.normal(0.0, w_sigma, (64, 3, 7, 7)))
    g, b_ = r.normal(1.0, 0.1, 64), r.normal(0.0, 0.1, 64)
    var = 147 * 1.0 * w_sigma ** 2                 # image ~ N(0, 1), fp32 weights
    inv = g / np.sqrt(var + 1e-5)                  # BN follows the 3x3 max pool
    out["stem"] = dict(w=sw, scale=f32(inv), shift=f32(b_ - inv * POOL_MEAN[9] * np.sqrt(var)))
    u = _units(bits_a) + _units(bits_w)

    def qconv(o, c, k):
        w = f32(r.normal(0.0, w_sigma, (o, c, k, k)))
        ws = weight_prescale(w, bits_w)
        scale, shift = bn_affine(r, o, c * k * k, bits_a, bits_w, ws, u, w_ms=weight_ms(w, ws, bits_w))
        return dict(w=w, w_scale=ws, scale=scale, shift=shift, k=k)

    blocks = []
    c_in = 64
    for stage, width in enumerate((64, 128, 256, 512)):
        for j in range(2):
            stride = 2 if (stage > 0 and j == 0) else 1
            blk = dict(stride=stride, c1=qconv(width, c_in, 3), c2=qconv(width, width, 3),
                       down=qconv(width, c_in, 1) if stride == 2 else None)
            blocks.append(blk)
            c_in = width
    out["blocks"] = blocks
    fw = f32(r.normal(0.0, w_sigma, (classes, 512)))
    g, b_ = r.normal(1.0, 0.1, classes), r.normal(0.0, 0.1, classes)
    var = 512 * _LEVEL_MS[bits_a] * w_sigma ** 2
    out["fc"] = dict(w=fw, scale=f32(g / np.sqrt(var + 1e-5)), shift=f32(b_))
    return out


# Second moment of a HardTanh output of a unit-variance input (the activations
# the weight-only blocks consume); used only to size the synthetic BN maps.
_HARDTANH_MS = 0.6


def wresnet_params(seed, n=18, bits_w=3, classes=10, hw=32, w_sigma=0.05):
    """Weight-only MINW-Net residual network of Table III (CIFAR ResNet-(6n+2),
    ResNet-110 for n = 18): an fp32 3x3 stem 3 -> 16 (fp32 weights), three
    stages of n basic blocks with 16, 32 and 64 channels (stride 2 and a 1x1
    shortcut entering stages 2 and 3) whose weights are quantized to N-bit
    levels while the activations stay full precision, and an fp32 classifier.
    Latent weights ~ N(0, w_sigma); synthetic BN maps sized from the input and
    level second moments (the block convolutions' outputs are in level
    units)."""
    r = rng(seed)
    out = dict(n=n, bits_w=bits_w, thr_w=DEFAULT_THR[bits_w], classes=classes, hw=hw)
    sw = f32(r.normal(0.0, w_sigma, (16, 3, 3, 3)))
    g, b_ = r.normal(1.0, 0.1, 16), r.normal(0.0, 0.1, 16)
    var = 27 * _LEVEL_MS[0] * w_sigma ** 2         # images U(-1, 1), fp32 weights
    out["stem"] = dict(w=sw, scale=f32(g / np.sqrt(var + 1e-5)), shift=f32(b_))
    unit2 = 4.0 ** _units(bits_w)

    def wconv(o, c, k):
        w = f32(r.normal(0.0, w_sigma, (o, c, k, k)))
        ws = weight_prescale(w, bits_w)
        gg, bb = r.normal(1.0, 0.1, o), r.normal(0.0, 0.1, o)
        v = c * k * k * _HARDTANH_MS * weight_ms(w, ws, bits_w) * unit2
        return dict(w=w, w_scale=ws, scale=f32(gg / np.sqrt(v + 1e-5)), shift=f32(bb), k=k)

    blocks = []
    c_in = 16
    for stage, width in enumerate((16, 32, 64)):
        for j in range(n):
            stride = 2 if (stage > 0 and j == 0) else 1
            blocks.append(dict(stride=stride, c1=wconv(width, c_in, 3), c2=wconv(width, width, 3),
                               down=wconv(width, c_in, 1) if stride == 2 else None))
            c_in = width
    out["blocks"] = blocks
    fw = f32(r.normal(0.0, w_sigma, (classes, 64)))
    g, b_ = r.normal(1.0, 0.1, classes), r.normal(0.0, 0.1, classes)
    var = 64 * _HARDTANH_MS * w_sigma ** 2
    out["fc"] = dict(w=fw, scale=f32(g / np.sqrt(var + 1e-5)), shift=f32(b_))
    return out


def wresnet_input(seed, B, hw=32):
    """CIFAR-shaped synthetic images, U(-1, 1)."""
    return f32(rng(seed).uniform(-1.0, 1.0, (B, 3, hw, hw)))


def wdense_params(seed, layers=16, growth=12, bits_w=3, classes=10, hw=32, w_sigma=0.05):
    """Weight-only MINW-Net DenseNet-BC of Table III (DenseNet-100 for
    layers = 16, growth 12): an fp32 3x3 stem 3 -> 2 growth (fp32 weights),
    three dense blocks of ``layers`` bottleneck layers (1x1 conv to 4 growth
    channels, then 3x3 conv to growth channels, each with its BN and
    HardTanh, concatenated onto the block's features), transitions with
    compression 1/2 (1x1 conv, BN, HardTanh, 2x2 average pool), and an fp32
    classifier.  Latent weights ~ N(0, w_sigma); BN maps as wresnet_params."""
    r = rng(seed)
    k = growth
    out = dict(layers=layers, growth=k, bits_w=bits_w, thr_w=DEFAULT_THR[bits_w], classes=classes, hw=hw)
    c0 = 2 * k
    sw = f32(r.normal(0.0, w_sigma, (c0, 3, 3, 3)))
    g, b_ = r.normal(1.0, 0.1, c0), r.normal(0.0, 0.1, c0)
    var = 27 * _LEVEL_MS[0] * w_sigma ** 2
    out["stem"] = dict(w=sw, scale=f32(g / np.sqrt(var + 1e-5)), shift=f32(b_))
    unit2 = 4.0 ** _units(bits_w)

    def wconv(o, c, kk):
        w = f32(r.normal(0.0, w_sigma, (o, c, kk, kk)))
        ws = weight_prescale(w, bits_w)
        gg, bb = r.normal(1.0, 0.1, o), r.normal(0.0, 0.1, o)
        v = c * kk * kk * _HARDTANH_MS * weight_ms(w, ws, bits_w) * unit2
        return dict(w=w, w_scale=ws, scale=f32(gg / np.sqrt(v + 1e-5)), shift=f32(bb), k=kk)

    blocks, trans = [], []
    c = c0
    for blk in range(3):
        lay = []
        for _ in range(layers):
            lay.append(dict(b=wconv(4 * k, c, 1), c=wconv(k, 4 * k, 3)))
            c += k
        blocks.append(lay)
        if blk < 2:
            trans.append(wconv(c // 2, c, 1))
            c //= 2
    out["blocks"], out["trans"] = blocks, trans
    fw = f32(r.normal(0.0, w_sigma, (classes, c)))
    g, b_ = r.normal(1.0, 0.1, classes), r.normal(0.0, 0.1, classes)
    var = c * _HARDTANH_MS * w_sigma ** 2
    out["fc"] = dict(w=fw, scale=f32(g / np.sqrt(var + 1e-5)), shift=f32(b_))
    out["features"] = c
    return out


def resnet18_input(seed, B, hw=224):
    """ImageNet-shaped synthetic images, N(0, 1)."""
    return f32(rng(seed).standard_normal((B, 3, hw, hw)))
