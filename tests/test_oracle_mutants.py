"""The oracle's pins against planted mistakes: for each plausible mistake in
an oracle function (a dropped term, a wrong sign, bound, index or operand
order, an extra rounding), a copy of the function with that mistake is put in
the oracle's place, on the CPU, and at least one committed pin must fail on
it.  A mistake no pin catches would pass unnoticed into every parity test
that uses the oracle as its reference."""
import numpy as np
import pytest

from oracle import network as N
from oracle import oracle as O
from paper_2003_04296_gb300.inputs import DEFAULT_THR
import tests.test_oracle_aqe as TA
import tests.test_oracle_epilogue as TE
import tests.test_oracle_levels as TL
import tests.test_oracle_network as TN
import tests.test_oracle_pack_conv as TP
import tests.test_oracle_train as TT
import tests.test_oracle_wdense as TD
import tests.test_oracle_wonly as TW
import tests.test_oracle_wresnet as TR

# the oracle's own functions, kept before any patch
_h, _quantize, _aqe_f, _aqe_b = O.h, O.quantize, O.aqe_forward, O.aqe_backward
_pack, _conv, _conv_real = O.pack, O.conv2d_levels, O.conv2d_real
_avg, _avg2, _fc_step = O.avgpool_f32, N.avgpool2_f32, O.fc_train_step
_linear, _maxpool, _igrad, _wgrad = O.linear_f32_seq, O.maxpool_f32, O.conv2d_input_grad, O.conv2d_weight_grad
_stoch = O.aqe_forward_stochastic
_convnet_layer = N.convnet_layer
_maxpool_i32 = O.maxpool_i32


def _pins_of(mod, name, params):
    fn = getattr(mod, name)
    return [lambda p=p: fn(*p) for p in params]


GOLDEN_LEVELS = _pins_of(TL, "test_golden_levels", TL._golden_rows())
GOLDEN_PACK = _pins_of(TP, "test_pack_golden", TP._golden())


# ---------------------------------------------------------------- mutants --

def h_sign_of_zero(x, bits, thr=None, scale=1.0):
    """Eq. sign read as +1 at zero."""
    v = _h(x, bits, thr, scale)
    return 1.0 if bits == 1 and np.float32(x) == 0 else v


def h_strict_thresholds(x, bits, thr=None, scale=1.0):
    """Eq. tnn / qnn with < in place of <=: a value on a threshold steps up."""
    t = [np.float32(v) for v in (thr if thr is not None else DEFAULT_THR[bits]) if v > 0]
    u = np.float32(np.float32(x) * np.float32(scale))
    if bits > 1 and abs(u) in t:
        return _h(np.nextafter(u, np.float32(np.inf) * np.sign(u)), bits, thr, 1.0)
    return _h(x, bits, thr, scale)


def quantize_half_steps(x, bits, thr=None, scale=None):
    """3-bit levels spaced by 1/3 instead of powers of two."""
    lv = _quantize(x, bits, thr, scale)
    if bits == 3:
        lv = np.where(np.abs(lv) == 0.25, np.sign(lv) / 3, lv)
    return lv


def aqe_forward_swapped(x, alpha, bits, thr=None, scale=1.0):
    """alpha and 1 - alpha exchanged in Eq. ours."""
    return _aqe_f(x, 1.0 - alpha, bits, thr, scale)


def aqe_forward_no_residual(x, alpha, bits, thr=None, scale=1.0):
    """Eq. ours without its (1 - alpha) a term."""
    x = np.asarray(x, dtype=np.float32)
    return alpha * _quantize(x.reshape(1, -1), bits, thr)[0].reshape(x.shape)


def aqe_backward_alpha(x, g, alpha):
    """Eq. activation with factor alpha in place of 2 alpha."""
    return _aqe_b(x, g, alpha) / 2


def aqe_backward_open(x, g, alpha):
    """The mask 1[|a| < 1] in place of 1[|a| <= 1]."""
    gx = _aqe_b(x, g, alpha)
    return np.where(np.abs(np.asarray(x, dtype=np.float32)) == 1.0, 0.0, gx)


def pack_msb_first(levels, bits):
    """Channel c at bit 31 - c % 32 instead of bit c % 32."""
    w = _pack(levels, bits)
    out = np.zeros_like(w)
    for b in range(32):
        out |= ((w >> np.uint32(b)) & np.uint32(1)) << np.uint32(31 - b)
    return out


def pack_planes_swapped(levels, bits):
    """Planes in reverse order (magnitude before sign)."""
    return np.ascontiguousarray(_pack(levels, bits)[..., ::-1, :])


def conv_flipped(a_lv, w_lv, stride, pad, bits_a, bits_w):
    """A true convolution (flipped taps) in place of the correlation."""
    return _conv(a_lv, np.ascontiguousarray(np.asarray(w_lv)[:, :, ::-1, ::-1]), stride, pad, bits_a, bits_w)


def conv_taps_transposed(a_lv, w_lv, stride, pad, bits_a, bits_w):
    """ky and kx exchanged."""
    return _conv(a_lv, np.ascontiguousarray(np.asarray(w_lv).transpose(0, 1, 3, 2)), stride, pad, bits_a, bits_w)


def affine_two_roundings(acc, scale, shift):
    """BN as an fp32 multiply, rounded, then an fp32 add."""
    s = np.asarray(scale, dtype=np.float32).reshape((1, -1) + (1,) * (acc.ndim - 2))
    t = np.asarray(shift, dtype=np.float32).reshape(s.shape)
    return ((acc.astype(np.float32) * s).astype(np.float32) + t).astype(np.float32)


def hardtanh_relu(y):
    """A clamp to [0, 1] in place of [-1, 1]."""
    return np.clip(np.asarray(y, dtype=np.float32), 0.0, 1.0)


def conv_seq_tap_major(x, w, stride, pad):
    """The fp32 chain over (ky, kx, ci) instead of (ci, ky, kx)."""
    x, w = np.asarray(x, dtype=np.float32), np.asarray(w, dtype=np.float32)
    B, C, H, W = x.shape
    O_, _, kh, kw = w.shape
    Ho, Wo = (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1
    out = np.zeros((B, O_, Ho, Wo), dtype=np.float32)
    for b in range(B):
        for o in range(O_):
            for y in range(Ho):
                for xx in range(Wo):
                    s = np.float32(0)
                    for ky in range(kh):
                        for kx in range(kw):
                            for c in range(C):
                                yi, xi = y * stride - pad + ky, xx * stride - pad + kx
                                if 0 <= yi < H and 0 <= xi < W:
                                    s = np.float32(s + np.float32(x[b, c, yi, xi] * w[o, c, ky, kx]))
                    out[b, o, y, xx] = s
    return out


def bf16_truncate(x):
    """bf16 by dropping the low 16 bits (no rounding)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) & np.uint32(0xFFFF0000)
    return u.view(np.float32)


def conv_real_flipped(a, w, stride, pad):
    """The real-valued convolution with flipped taps."""
    return _conv_real(a, np.ascontiguousarray(np.asarray(w)[:, :, ::-1, ::-1]), stride, pad)


def sgd_no_clip(w, g, lr):
    """The update without its clip to [-1, 1]."""
    return (np.asarray(w, dtype=np.float32) - np.float32(lr) * np.asarray(g, dtype=np.float32)).astype(np.float32)


def avgpool_wrong_count(x):
    """The global average divided by one pixel fewer."""
    x = np.asarray(x, dtype=np.float32)
    hw = x.shape[2] * x.shape[3]
    return (_avg(x).astype(np.float64) * hw / (hw - 1)).astype(np.float32)


def avgpool2_shifted(t):
    """The 2x2 windows taken one column to the right (wrapping)."""
    return _avg2(np.roll(np.asarray(t, dtype=np.float32), -1, axis=3))


def linear_bias_first(x, w, bias=None):
    """The fully connected layer's chain started from the bias instead of
    adding it last (each step x w + s in fp64, rounded to fp32)."""
    x, w = np.asarray(x, dtype=np.float32), np.asarray(w, dtype=np.float32)
    y = np.empty((x.shape[0], w.shape[0]), dtype=np.float32)
    for i in range(x.shape[0]):
        for o in range(w.shape[0]):
            acc = np.float32(0.0 if bias is None else bias[o])
            for k in range(x.shape[1]):
                acc = np.float32(float(x[i, k]) * float(w[o, k]) + float(acc))
            y[i, o] = acc
    return y


def maxpool_shifted(x, k, s, p):
    """The pooling windows one column off."""
    return _maxpool(np.roll(np.asarray(x, dtype=np.float32), 1, axis=3), k, s, p)


def input_grad_flipped(g, w, stride, pad, H, W):
    """The input gradient with unflipped taps (a correlation with W in place of its transpose)."""
    return _igrad(g, np.ascontiguousarray(np.asarray(w)[:, :, ::-1, ::-1]), stride, pad, H, W)


def weight_grad_flipped(g, a, kh, kw, stride, pad):
    """The weight gradient with its taps reversed."""
    return np.ascontiguousarray(_wgrad(g, a, kh, kw, stride, pad)[:, :, ::-1, ::-1])


def stochastic_halves_swapped(x, alpha, seed, offset=0):
    """The stochastic AQE drawing each 64-bit word's high half first."""
    _, z = _stoch(x, alpha, seed, offset)
    z = np.asarray(z).copy()
    n2 = z.size // 2 * 2
    z[:n2] = z[:n2].reshape(-1, 2)[:, ::-1].ravel()
    xd = np.asarray(x, dtype=np.float32).astype(np.float64)
    s = np.where(xd - z.astype(np.float64) > 0, 1.0, -1.0)
    return alpha * s + (1.0 - alpha) * xd, z


def quantize_divided_scale(x, bits, thr=None, scale=None):
    """The per-channel prescale (R7) applied as a division."""
    if scale is None:
        return _quantize(x, bits, thr, None)
    return _quantize(x, bits, thr, (1.0 / np.asarray(scale, dtype=np.float64)).astype(np.float32))


def maxpool_i32_shifted(acc, k=2, s=2):
    """The integer pooling windows one row down (wrapping)."""
    return _maxpool_i32(np.roll(np.asarray(acc), -1, axis=2), k, s)


def conv_units_doubled(a_lv, w_lv, stride, pad, bits_a, bits_w):
    """3-bit levels counted in units of 1/2 instead of 1/4 (a wrong integer scale)."""
    acc = _conv(a_lv, w_lv, stride, pad, bits_a, bits_w)
    return acc // 2 if 3 in (bits_a, bits_w) else acc


def convnet_layer_hwc_flatten(layer, a, thr_a, thr_w):
    """The first fully connected layer flattening its input in (h, w, c)
    order instead of R14's (c, h, w)."""
    if layer["kind"] != "conv" and layer["bits_in"] != 0 and np.ndim(a) == 4:
        a = np.ascontiguousarray(np.asarray(a).transpose(0, 2, 3, 1)).reshape(np.shape(a))
    return _convnet_layer(layer, a, thr_a, thr_w)


def wconv_no_bf16(conv, a, stride, bits_w, thr_w):
    """A weight-only convolution that reads its fp32 input without the bf16 rounding (R19)."""
    k = conv["w"].shape[2]
    acc = O.conv2d_real(np.asarray(a, dtype=np.float64), N._wlevels(conv, bits_w, thr_w), stride, k // 2)
    return O.affine(acc.astype(np.float32), conv["scale"], conv["shift"])


def wdense_layer_no_hardtanh(lay, F, bits_w, thr_w):
    """The 3x3's HardTanh dropped."""
    h = O.hardtanh(N.wconv(lay["b"], F, 1, bits_w, thr_w))
    return h, O.bf16_round(N.wconv(lay["c"], h, 1, bits_w, thr_w))


def wdense_transition_pool_first(conv, F, bits_w, thr_w):
    """The pool taken before the HardTanh."""
    return O.bf16_round(O.hardtanh(_avg2(N.wconv(conv, F, 1, bits_w, thr_w))))


def wresnet_block_no_shortcut(blk, a, bits_w, thr_w):
    """The residual block without its shortcut."""
    h = O.hardtanh(N.wconv(blk["c1"], a, blk["stride"], bits_w, thr_w))
    return h, O.hardtanh(N.wconv(blk["c2"], h, 1, bits_w, thr_w))


def fc_step_unmasked_weights(A, W, G, alpha, lr, bits_w, thr_w, q_a=None, a_pre=None):
    """The weight step without the mask of Eq. weight (a plain STE)."""
    a_out, g_in, _, a_pre = _fc_step(A, W, G, alpha, lr, bits_w, thr_w, q_a, a_pre)
    g_t = G if q_a is None else O.aqe_backward_f32(a_pre, G, alpha)
    g_w = (np.asarray(g_t, dtype=np.float64).T @ np.asarray(A, dtype=np.float64)).astype(np.float32)
    return a_out, g_in, O.sgd_clip(W, g_w, lr), a_pre


MUTANTS = [
    ("h: sign(0) = +1", O, "h", h_sign_of_zero, GOLDEN_LEVELS),
    ("h: strict thresholds", O, "h", h_strict_thresholds,
     GOLDEN_LEVELS + _pins_of(TL, "test_threshold_neighbours", [(2,), (3,)])),
    ("quantize: 3-bit levels not powers of two", O, "quantize", quantize_half_steps,
     _pins_of(TL, "test_level_set_membership_and_monotone", [(3,)])),
    ("AQE forward: alpha swapped", O, "aqe_forward", aqe_forward_swapped,
     _pins_of(TA, "test_alpha_limits", [(1,), (2,), (3,)])),
    ("AQE forward: (1 - alpha) a dropped", O, "aqe_forward", aqe_forward_no_residual,
     _pins_of(TA, "test_alpha_limits", [(1,), (2,), (3,)])),
    ("AQE backward: factor alpha", O, "aqe_backward", aqe_backward_alpha,
     _pins_of(TA, "test_backward_matches_central_difference", [(0.5,)]) + [TA.test_half_alpha_is_ste]),
    ("AQE backward: open interval", O, "aqe_backward", aqe_backward_open, [TA.test_backward_mask_is_closed_interval]),
    ("pack: MSB first", O, "pack", pack_msb_first, GOLDEN_PACK),
    ("pack: planes reversed", O, "pack", pack_planes_swapped, GOLDEN_PACK),
    ("conv: flipped taps", O, "conv2d_levels", conv_flipped,
     _pins_of(TP, "test_conv_matches_torch_float64", [(1, 1, 1, 1, 3), (3, 3, 2, 1, 3)])),
    ("conv: ky and kx exchanged", O, "conv2d_levels", conv_taps_transposed,
     _pins_of(TP, "test_conv_matches_torch_float64", [(1, 1, 1, 1, 3), (2, 2, 2, 3, 7)])),
    ("BN: two roundings", O, "affine", affine_two_roundings, [TE.test_affine_is_single_rounding]),
    ("HardTanh: clamp to [0, 1]", O, "hardtanh", hardtanh_relu, [TE.test_hardtanh]),
    ("fp32 first layer: tap-major chain", O, "conv2d_f32_seq", conv_seq_tap_major,
     [TE.test_conv_f32_seq_order_and_bound]),
    ("bf16: truncation", O, "bf16_round", bf16_truncate, [TW.test_bf16_round_matches_torch]),
    ("real conv: flipped taps", O, "conv2d_real", conv_real_flipped,
     _pins_of(TW, "test_conv2d_real_matches_torch", [((2, 5, 7, 6, 4, 3, 1, 1),)])),
    ("update: no clip", O, "sgd_clip", sgd_no_clip, [TT.test_sgd_clip_single_rounding]),
    ("global average: wrong count", O, "avgpool_f32", avgpool_wrong_count, [TE.test_avgpool_and_linear_bounds]),
    ("2x2 average: shifted windows", N, "avgpool2_f32", avgpool2_shifted, [TD.test_avgpool2_against_numpy]),
    ("DenseNet layer: HardTanh dropped", N, "wdense_layer", wdense_layer_no_hardtanh,
     _pins_of(TD, "test_small_wdense", [(3,)])),
    ("DenseNet transition: pool first", N, "wdense_transition", wdense_transition_pool_first,
     _pins_of(TD, "test_small_wdense", [(3,)])),
    ("ResNet-110 block: shortcut dropped", N, "wresnet_block", wresnet_block_no_shortcut,
     _pins_of(TR, "test_small_wresnet_blocks", [(3,)])),
    ("training step: weight mask dropped", O, "fc_train_step", fc_step_unmasked_weights,
     _pins_of(TT, "test_fc_train_step_wiring", [(False,), (True,)])),
    ("fully connected: bias first", O, "linear_f32_seq", linear_bias_first, [TE.test_linear_and_avgpool_order]),
    ("max pool: shifted windows", O, "maxpool_f32", maxpool_shifted, [TE.test_maxpool_f32_vs_torch]),
    ("input gradient: unflipped taps", O, "conv2d_input_grad", input_grad_flipped,
     _pins_of(TT, "test_conv_backward_products_match_autograd", [(1, 1, 3)]) + [TT.test_conv_train_step_gradients]),
    ("weight gradient: reversed taps", O, "conv2d_weight_grad", weight_grad_flipped,
     _pins_of(TT, "test_conv_backward_products_match_autograd", [(1, 1, 3)]) + [TT.test_conv_train_step_gradients]),
    ("stochastic AQE: high half first", O, "aqe_forward_stochastic", stochastic_halves_swapped,
     [TA.test_stochastic_noise_words_follow_r18, TA.test_noise_grid_and_uniformity,
      TA.test_stochastic_limits_and_counter_layout]),
    ("quantize: prescale divided", O, "quantize", quantize_divided_scale, [TL.test_per_channel_scale_quantize]),
    ("integer max pool: shifted windows", O, "maxpool_i32", maxpool_i32_shifted, [TE.test_maxpool_i32_vs_reshape]),
    ("conv: 3-bit units of 1/2", O, "conv2d_levels", conv_units_doubled,
     _pins_of(TP, "test_conv_matches_torch_float64", [(3, 1, 1, 1, 3), (1, 3, 1, 1, 3)])),
    ("ConvNet: flatten in (h, w, c) order", N, "convnet_layer", convnet_layer_hwc_flatten,
     _pins_of(TN, "test_small_convnet_layerwise", [(1, 1), (2, 2)])),
    ("weight-only conv: no bf16 input rounding", N, "wconv", wconv_no_bf16,
     _pins_of(TR, "test_small_wresnet_blocks", [(3,)]) + _pins_of(TD, "test_small_wdense", [(3,)])),
]


def test_pins_pass_on_the_oracle():
    """The harness itself: every pin used below passes on the unmodified oracle."""
    for _, _, _, _, pins in MUTANTS:
        for pin in pins:
            pin()


@pytest.mark.parametrize("name,module,attr,mutant,pins", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(monkeypatch, name, module, attr, mutant, pins):
    monkeypatch.setattr(module, attr, mutant)
    failed = 0
    for pin in pins:
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed > 0, f"no pin catches the mistake: {name}"
