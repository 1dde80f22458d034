"""Whole-network forward passes composed from the oracle's layer routines
(test infrastructure only).

MINW-Net inference (Algorithm 1, inference branch): for l = 1..n the weights
are quantized (W^ = h(W)), the layer computes a~_l = a^q_{l-1} W^_l, and every
layer but the last quantizes its output (a^q_l = h(a~_l)).  Around the product
sit the layer constructs of Sec. III-E: {QuantizedConv-pooling-BN-HardTanh}
or {QuantizedConv-BN-HardTanh}; the input of the first convolution stays
fp32 while its weights are quantized; batch normalisation also follows the
fully connected layers; the last layer's BN output is the fp32 logits.
"""
import numpy as np

from . import oracle as O


def _layer_levels_w(layer, thr_w):
    return O.quantize(layer["w"], layer["bits_w"], thr_w, layer["w_scale"])


def convnet_layer(layer, a, thr_a, thr_w):
    """One layer of the Model-A-shaped ConvNet.

    ``a`` is the fp32 image for the first layer and the previous layer's
    HardTanh output otherwise (its quantization h is applied here).  Returns
    (acc, y): the integer accumulator (None for the fp32 first layer, whose raw
    output is fp32) after pooling, and the layer's fp32 output after BN and,
    unless it is the last layer, HardTanh."""
    wl = _layer_levels_w(layer, thr_w)
    acc = None
    if layer["bits_in"] == 0:
        z = O.conv2d_f32_seq(a, wl.astype(np.float32), layer["stride"], layer["pad"])
        if layer["pool"]:
            z = O.maxpool_f32(z, 2, 2, 0)
        y = O.affine(z, layer["scale"], layer["shift"])
    else:
        al = O.quantize(a, layer["bits_in"], thr_a)
        if layer["kind"] == "conv":
            acc = O.conv2d_levels(al, wl, layer["stride"], layer["pad"],
                                  layer["bits_in"], layer["bits_w"])
            if layer["pool"]:
                acc = O.maxpool_i32(acc, 2, 2)
        else:
            B = al.shape[0]
            flat = al.reshape(B, -1)                       # (c, h, w) order
            acc = O.conv2d_levels(flat[:, :, None, None], wl[:, :, None, None], 1, 0,
                                  layer["bits_in"], layer["bits_w"])
            acc = acc.reshape(B, -1)
        y = O.affine(acc, layer["scale"], layer["shift"])
    if layer["bits_out"] != 0:
        y = O.hardtanh(y)
    return acc, y


def convnet_forward(net, x, keep=False):
    """Forward pass of the ConvNet built by ``inputs.convnet_params``.
    Returns the fp32 logits, and with ``keep`` also the per-layer (acc, y)."""
    a = x
    trace = []
    for layer in net["layers"]:
        acc, a = convnet_layer(layer, a, net["thr_a"], net["thr_w"])
        if keep:
            trace.append((acc, a))
    return (a, trace) if keep else a


def activation_levels(y, bits, thr):
    """Quantized levels h(y) of a layer output (what the next layer consumes)."""
    return O.quantize(y, bits, thr)


def resnet18_forward(net, x, keep=False):
    """Forward pass of the ResNet-18-shaped MINW-Net built by
    ``inputs.resnet18_params``.  The paper leaves the residual wiring open;
    the reading followed (one fp32 operation per written step):
      stem : fp32 7x7/2 conv (fp32 weights, pad 3) -> 3x3/2 max pool (pad 1)
             -> BN -> HardTanh -> h  (the block order of Sec. III-E)
      block: u = h(x); v = h(HardTanh(BN1(conv1(u))));
             y = BN2(conv2(v)) + s, s = u or BN_d(conv_d(u)) (1x1 / 2);
             next input = HardTanh(y) (quantized by the next block's h)
      head : global average pool of h(last output) -> fp32 FC -> BN."""
    ba, bw = net["bits_a"], net["bits_w"]
    ta, tw = net["thr_a"], net["thr_w"]
    st = net["stem"]
    z = O.conv2d_f32_seq(x, st["w"], 2, 3)
    z = O.maxpool_f32(z, 3, 2, 1)
    a = O.hardtanh(O.affine(z, st["scale"], st["shift"]))
    trace = [a]
    for blk in net["blocks"]:
        u = O.quantize(a, ba, ta)
        c1, c2 = blk["c1"], blk["c2"]
        w1 = O.quantize(c1["w"], bw, tw, c1["w_scale"])
        acc1 = O.conv2d_levels(u, w1, blk["stride"], 1, ba, bw)
        v = O.quantize(O.hardtanh(O.affine(acc1, c1["scale"], c1["shift"])), ba, ta)
        w2 = O.quantize(c2["w"], bw, tw, c2["w_scale"])
        y = O.affine(O.conv2d_levels(v, w2, 1, 1, ba, bw), c2["scale"], c2["shift"])
        if blk["down"] is None:
            s = u.astype(np.float32)
        else:
            d = blk["down"]
            wd = O.quantize(d["w"], bw, tw, d["w_scale"])
            s = O.affine(O.conv2d_levels(u, wd, 2, 0, ba, bw), d["scale"], d["shift"])
        a = O.hardtanh((y + s).astype(np.float32))
        trace.append(a)
    last = O.quantize(a, ba, ta).astype(np.float32)
    pooled = O.avgpool_f32(last)
    fc = net["fc"]
    logits = O.affine(O.linear_f32_seq(pooled, fc["w"]), fc["scale"], fc["shift"])
    return (logits, trace) if keep else logits


def _wlevels(conv, bits_w, thr_w):
    """A weight-only layer's weights: the levels of h in integer units
    (quarters for 3-bit), exact in bf16."""
    return O.quantize(conv["w"], bits_w, thr_w, conv["w_scale"]) * 2.0 ** O.units_shift(bits_w)


def wconv(conv, a, stride, bits_w, thr_w):
    """One weight-only convolution with its BN (the SHIFT ADDER layer of
    Sec. IV): the fp32 activation rounded to bf16 (the layer's 16-bit input),
    the product with the weight levels summed in fp64 and rounded to fp32,
    then the BN map (fmaf).  Returns the fp32 BN output."""
    k = conv["w"].shape[2]
    ab = O.bf16_round(a).astype(np.float64)
    acc = O.conv2d_real(ab, _wlevels(conv, bits_w, thr_w), stride, k // 2)
    return O.affine(acc.astype(np.float32), conv["scale"], conv["shift"])


def wresnet_block(blk, a, bits_w, thr_w):
    """One block of the weight-only residual network: h = HardTanh(BN1(conv1(a))),
    out = HardTanh(BN2(conv2(h)) + s), s = a or BN_d(conv_d(a)) (one fp32 add).
    Returns (h, out)."""
    h = O.hardtanh(wconv(blk["c1"], a, blk["stride"], bits_w, thr_w))
    y2 = wconv(blk["c2"], h, 1, bits_w, thr_w)
    s = a if blk["down"] is None else wconv(blk["down"], a, 2, bits_w, thr_w)
    return h, O.hardtanh((y2 + s).astype(np.float32))


def wresnet_head(net, a):
    """Global average pool (one fp32 sum in pixel order, one division), the
    fp32 fully connected layer (one fmaf chain) and its BN: the logits."""
    fc = net["fc"]
    return O.affine(O.linear_f32_seq(O.avgpool_f32(a), fc["w"]), fc["scale"], fc["shift"])


def wresnet_forward(net, x, keep=False):
    """Forward pass of the weight-only residual network of Table III built by
    ``inputs.wresnet_params`` (a CIFAR ResNet-(6n+2), ResNet-110 for n = 18).
    The paper leaves the wiring open; the reading followed:
      stem : fp32 3x3 conv (fp32 weights, one fmaf chain per output) -> BN
             -> HardTanh
      block: wresnet_block; the stage entries (stride 2) take a 1x1 / 2
             shortcut with quantized weights
      head : wresnet_head.
    With ``keep`` also returns every block's output (after the stem first)."""
    bw, tw = net["bits_w"], net["thr_w"]
    st = net["stem"]
    a = O.hardtanh(O.affine(O.conv2d_f32_seq(x, st["w"], 1, 1), st["scale"], st["shift"]))
    trace = [a]
    for blk in net["blocks"]:
        _, a = wresnet_block(blk, a, bw, tw)
        trace.append(a)
    logits = wresnet_head(net, a)
    return (logits, trace) if keep else logits


def avgpool2_f32(t):
    """2x2 / 2 average pool of fp32 [B][C][H][W]: ((t00 + t01) + t10) + t11 in
    fp32, then times 1/4 (exact)."""
    t = np.asarray(t, dtype=np.float32)
    s = (t[:, :, 0::2, 0::2] + t[:, :, 0::2, 1::2]).astype(np.float32)
    s = (s + t[:, :, 1::2, 0::2]).astype(np.float32)
    s = (s + t[:, :, 1::2, 1::2]).astype(np.float32)
    return (s * np.float32(0.25)).astype(np.float32)


def wdense_layer(lay, F, bits_w, thr_w):
    """One bottleneck layer of the weight-only DenseNet: h = HardTanh(BN(conv
    1x1(F))), n = HardTanh(BN(conv 3x3(h))); returns (h, bf16(n)), the new
    features in the 16-bit form the block holds them in."""
    h = O.hardtanh(wconv(lay["b"], F, 1, bits_w, thr_w))
    n = O.hardtanh(wconv(lay["c"], h, 1, bits_w, thr_w))
    return h, O.bf16_round(n)


def wdense_transition(conv, F, bits_w, thr_w):
    """Transition: bf16(avgpool 2x2(HardTanh(BN(conv 1x1(F)))))."""
    t = O.hardtanh(wconv(conv, F, 1, bits_w, thr_w))
    return O.bf16_round(avgpool2_f32(t))


def wdense_forward(net, x, keep=False):
    """Forward pass of the weight-only DenseNet-BC of Table III built by
    ``inputs.wdense_params`` (DenseNet-100 for 16 layers per block, growth
    12).  The paper gives no wiring beyond DenseNet's; the reading followed
    (the block order of Sec. III-E, conv -> BN -> HardTanh, in place of
    DenseNet's pre-activation):
      stem : fp32 3x3 conv (fp32 weights) -> BN -> HardTanh
      block: features F, held as bf16 (the form every convolution reads); each
             layer appends wdense_layer's growth channels
      trans: wdense_transition (channels halved, 2x2 average pool)
      head : global average pool of the last F (one fp32 sum in pixel order,
             one division) -> fp32 FC -> BN.
    With ``keep`` also returns each block's final features (bf16 values)."""
    bw, tw = net["bits_w"], net["thr_w"]
    st = net["stem"]
    F = O.bf16_round(O.hardtanh(O.affine(O.conv2d_f32_seq(x, st["w"], 1, 1), st["scale"], st["shift"])))
    finals = []
    for bi, lay_list in enumerate(net["blocks"]):
        for lay in lay_list:
            _, nb = wdense_layer(lay, F, bw, tw)
            F = np.concatenate([F, nb], axis=1)
        finals.append(F)
        if bi < len(net["trans"]):
            F = wdense_transition(net["trans"][bi], F, bw, tw)
    logits = wresnet_head(net, F)
    return (logits, finals) if keep else logits
