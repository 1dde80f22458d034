"""ctypes binding of libminw.so (include/minw.h).

Argument marshalling only: every function passes device pointers, sizes and
the current CUDA stream to the C entry point of the same name and raises on a
non-OK status.  Every step of the computation runs in the library's CUDA
kernels; there is no fallback of any kind.  torch provides device memory and
streams.
"""
import ctypes
import os

import torch

from . import build as _build

_LIB = None

MINW_OK, MINW_EINVAL, MINW_EUNSUPPORTED, MINW_ECUDA, MINW_ETIMEOUT, MINW_EDEVICE = range(6)
VARIANT_AUTO, VARIANT_POPC, VARIANT_TC, VARIANT_TC_E4M3, VARIANT_TC_E2M1, VARIANT_TC_E2M1_PAIRS = 0, 1, 2, 3, 4, 5
VARIANT_TC_E2M1_N128 = 6
CODES_E4M3, CODES_E2M1 = 0, 1
LAYER_CONV, LAYER_FC = 0, 1


class MinwError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


class Quant(ctypes.Structure):
    _fields_ = [("bits", ctypes.c_int32), ("thr", ctypes.c_float * 3), ("scale", ctypes.c_float)]


class BlockExtra(ctypes.Structure):
    _fields_ = [("res_codes", ctypes.c_void_p), ("res_bits", ctypes.c_int32), ("res_f32", ctypes.c_void_p),
                ("y_nhwc", ctypes.c_void_p), ("in_format", ctypes.c_int32), ("out_format", ctypes.c_int32),
                ("res_format", ctypes.c_int32), ("acc_out", ctypes.c_void_p), ("e2m1_pairs", ctypes.c_int32)]


class PlanOptions(ctypes.Structure):
    _fields_ = [("cta_pairs", ctypes.c_int32), ("channel_major", ctypes.c_int32),
                ("channel_major_min_tiles_per_sm", ctypes.c_int32), ("dup_weights", ctypes.c_int32),
                ("kblocks_per_stage", ctypes.c_int32), ("first_tma", ctypes.c_int32), ("pdl", ctypes.c_int32),
                ("graph", ctypes.c_int32), ("tma_lanes", ctypes.c_int32),
                ("resident_weights", ctypes.c_int32), ("first_tensor_cores", ctypes.c_int32),
                ("wait_cycles", ctypes.c_int64)]


STALL_CONV_TC, STALL_CONV_FIRST = 1, 2


class PipeRates(ctypes.Structure):
    _fields_ = [("sm_clock_mhz", ctypes.c_double), ("popc_per_s", ctypes.c_double),
                ("bmma_b1_mac_per_s", ctypes.c_double), ("imma_s8_mac_per_s", ctypes.c_double),
                ("tc_e4m3_flop_per_s", ctypes.c_double * 2), ("tc_e2m1_flop_per_s", ctypes.c_double * 2),
                ("tc_bf16_flop_per_s", ctypes.c_double * 2), ("tma_box_cycles", ctypes.c_double)]


class LayerDesc(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("C", ctypes.c_int32), ("H", ctypes.c_int32),
                ("W", ctypes.c_int32), ("O", ctypes.c_int32), ("kh", ctypes.c_int32),
                ("kw", ctypes.c_int32), ("stride", ctypes.c_int32), ("pad", ctypes.c_int32),
                ("pool", ctypes.c_int32), ("bits_in", ctypes.c_int32), ("bits_w", ctypes.c_int32),
                ("bits_out", ctypes.c_int32), ("thr_w", ctypes.c_float * 3),
                ("thr_out", ctypes.c_float * 3), ("w", ctypes.c_void_p), ("w_scale", ctypes.c_void_p),
                ("scale", ctypes.c_void_p), ("shift", ctypes.c_void_p), ("variant", ctypes.c_int32)]


WRESNET_MAX_N = 18
_NB = 3 * WRESNET_MAX_N


class WResNetDesc(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("bits_w", ctypes.c_int32), ("thr_w", ctypes.c_float * 3),
                ("image_hw", ctypes.c_int32), ("num_classes", ctypes.c_int32),
                ("stem_w", ctypes.c_void_p), ("stem_scale", ctypes.c_void_p), ("stem_shift", ctypes.c_void_p),
                ("c1_w", ctypes.c_void_p * _NB), ("c1_wscale", ctypes.c_void_p * _NB),
                ("c1_scale", ctypes.c_void_p * _NB), ("c1_shift", ctypes.c_void_p * _NB),
                ("c2_w", ctypes.c_void_p * _NB), ("c2_wscale", ctypes.c_void_p * _NB),
                ("c2_scale", ctypes.c_void_p * _NB), ("c2_shift", ctypes.c_void_p * _NB),
                ("down_w", ctypes.c_void_p * 2), ("down_wscale", ctypes.c_void_p * 2),
                ("down_scale", ctypes.c_void_p * 2), ("down_shift", ctypes.c_void_p * 2),
                ("fc_w", ctypes.c_void_p), ("fc_scale", ctypes.c_void_p), ("fc_shift", ctypes.c_void_p),
                ("keep_activations", ctypes.c_int32)]


WDENSE_MAX_LAYERS = 32
_NL = 3 * WDENSE_MAX_LAYERS


class WDenseDesc(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_int32), ("growth", ctypes.c_int32), ("bits_w", ctypes.c_int32),
                ("thr_w", ctypes.c_float * 3), ("image_hw", ctypes.c_int32), ("num_classes", ctypes.c_int32),
                ("stem_w", ctypes.c_void_p), ("stem_scale", ctypes.c_void_p), ("stem_shift", ctypes.c_void_p),
                ("b_w", ctypes.c_void_p * _NL), ("b_wscale", ctypes.c_void_p * _NL),
                ("b_scale", ctypes.c_void_p * _NL), ("b_shift", ctypes.c_void_p * _NL),
                ("c_w", ctypes.c_void_p * _NL), ("c_wscale", ctypes.c_void_p * _NL),
                ("c_scale", ctypes.c_void_p * _NL), ("c_shift", ctypes.c_void_p * _NL),
                ("t_w", ctypes.c_void_p * 2), ("t_wscale", ctypes.c_void_p * 2),
                ("t_scale", ctypes.c_void_p * 2), ("t_shift", ctypes.c_void_p * 2),
                ("fc_w", ctypes.c_void_p), ("fc_scale", ctypes.c_void_p), ("fc_shift", ctypes.c_void_p)]


class ResNet18Desc(ctypes.Structure):
    _fields_ = [("bits_a", ctypes.c_int32), ("bits_w", ctypes.c_int32), ("thr_a", ctypes.c_float * 3),
                ("thr_w", ctypes.c_float * 3), ("image_hw", ctypes.c_int32), ("num_classes", ctypes.c_int32),
                ("stem_w", ctypes.c_void_p), ("stem_scale", ctypes.c_void_p), ("stem_shift", ctypes.c_void_p),
                ("conv_w", ctypes.c_void_p * 16), ("conv_wscale", ctypes.c_void_p * 16),
                ("conv_scale", ctypes.c_void_p * 16), ("conv_shift", ctypes.c_void_p * 16),
                ("down_w", ctypes.c_void_p * 3), ("down_wscale", ctypes.c_void_p * 3),
                ("down_scale", ctypes.c_void_p * 3), ("down_shift", ctypes.c_void_p * 3),
                ("fc_w", ctypes.c_void_p), ("fc_scale", ctypes.c_void_p), ("fc_shift", ctypes.c_void_p)]


# name -> (restype, argtypes)
_P, _I32, _I64, _F = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
_QP = ctypes.POINTER(Quant)
SIGNATURES = {
    "minw_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "minw_version": (_I32, []),
    "aqe_forward": (ctypes.c_int, [_P, _P, _I64, _F, _QP, _P]),
    "aqe_backward": (ctypes.c_int, [_P, _P, _P, _I64, _F, _P]),
    "aqe_forward_stochastic": (ctypes.c_int, [_P, _P, _I64, _F, ctypes.c_uint64, ctypes.c_uint64, _P]),
    "minw_to_bf16_nhwc": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _P, _P]),
    "minw_to_bf16_nhwc_pad": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _P]),
    "minw_pack_weight_bf16_pad": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _QP, _P, _P, _P]),
    "minw_pack_weight_bf16": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _P, _P]),
    "minw_conv2d_bf16": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32, _I32, _I32,
                                        _I32, _P, _P, _P, _P]),
    "minw_conv2d_bf16_hardtanh": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32, _I32,
                                                 _I32, _P, _P, _P, _I32, _I32, _P, _P, _P]),
    "minw_bf16_matrix": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _P, _P]),
    "minw_sgd_clip": (ctypes.c_int, [_P, _P, _I64, _F, _P]),
    "minw_fc_train_workspace_bytes": (ctypes.c_size_t, [_I32, _I32, _I32]),
    "minw_conv_train_workspace_bytes": (ctypes.c_size_t, [_I32] * 9),
    "minw_conv_train_step": (ctypes.c_int, [_P, _P, _P] + [_I32] * 9 + [_F, _F, _QP, _QP, _P, _P, _P, _P,
                                            ctypes.c_size_t, _P]),
    "minw_fc_train_step": (ctypes.c_int, [_P, _P, _P, _I32, _I32, _I32, _F, _F, _QP, _QP, _P, _P, _P, _P,
                                          ctypes.c_size_t, _P]),
    "aqe_quantize_pack": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _F, _P, _P, _P]),
    "aqe_backward_masked": (ctypes.c_int, [_P, _P, _P, _I64, _F, _P]),
    "minw_pack_weights": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _P, _P]),
    "minw_conv2d": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32,
                                   _I32, _I32, _P, _P, _P, _P, _I32, _P]),
    "minw_conv_block": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32,
                                       _I32, _I32, _I32, _P, _P, _QP, _P, _P, _I32, _P]),
    "minw_conv_first": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32, _I32,
                                       _QP, _P, _I32, _P, _P, _QP, _P, _P, _P]),
    "aqe_quantize_codes": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _P]),
    "minw_pack_weight_codes": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _P, _P]),
    "aqe_quantize_codes_e2m1": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _P]),
    "minw_pack_weight_codes_e2m1": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _QP, _P, _P, _P]),
    "minw_conv2d_codes": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32,
                                         _I32, _I32, _P, _P, _P, _P, _P]),
    "minw_conv_block_codes": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32,
                                             _I32, _I32, _I32, _P, _P, _QP, _P, _P, _P, _P]),
    "minw_conv_block_codes_ex": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _I32, _I32,
                                                _I32, _I32, _I32, _P, _P, _QP, _P, _P, _P,
                                                ctypes.POINTER(BlockExtra), _P]),
    "minw_fc_workspace_bytes": (ctypes.c_size_t, [_I32, _I32, _I32]),
    "minw_fc_ksplit": (_I32, [_I32, _I32, _I32, ctypes.c_size_t]),
    "minw_get_plan_options": (ctypes.c_int, [ctypes.POINTER(PlanOptions)]),
    "minw_set_plan_options": (ctypes.c_int, [ctypes.POINTER(PlanOptions)]),
    "minw_test_stall_next_launch": (ctypes.c_int, [_I32]),
    "minw_measure_pipe_rates": (ctypes.c_int, [ctypes.POINTER(PipeRates), _P]),
    "minw_fc_codes": (ctypes.c_int, [_P, _I32, _I32, _I32, _P, _I32, _I32, _P, _P, _QP, _P, _P, _P, _P, _P,
                                     ctypes.c_size_t, _P]),
    "minw_fc_codes_noalloc": (ctypes.c_int, [_P, _I32, _I32, _I32, _P, _I32, _I32, _P, _P, _QP, _P, _P, _P, _P,
                                             _P]),
    "minw_net_create": (ctypes.c_int, [ctypes.POINTER(LayerDesc), _I32, _I32, _I32, _P,
                                       ctypes.POINTER(ctypes.c_void_p)]),
    "minw_resnet18_create": (ctypes.c_int, [ctypes.POINTER(ResNet18Desc), _I32, _P,
                                            ctypes.POINTER(ctypes.c_void_p)]),
    "minw_wresnet_create": (ctypes.c_int, [ctypes.POINTER(WResNetDesc), _I32, _P,
                                           ctypes.POINTER(ctypes.c_void_p)]),
    "minw_wresnet_activation": (ctypes.c_int, [_P, _I32, _P, ctypes.c_size_t, _P]),
    "minw_wdense_create": (ctypes.c_int, [ctypes.POINTER(WDenseDesc), _I32, _P, ctypes.POINTER(ctypes.c_void_p)]),
    "minw_wdense_features": (ctypes.c_int, [_P, _I32, _P, ctypes.c_size_t, ctypes.POINTER(ctypes.c_int32),
                                            ctypes.POINTER(ctypes.c_int32), _P]),
    "minw_forward": (ctypes.c_int, [_P, _P, _I32, _P, _P]),
    "minw_forward_host": (ctypes.c_int, [_P, _P, _I32, _P, _P]),
    "minw_net_enable_timing": (ctypes.c_int, [_P, _I32]),
    "minw_net_layer_times": (ctypes.c_int, [_P, _P]),
    "minw_net_layer_variants": (ctypes.c_int, [_P, _P]),
    "minw_net_layer_candidates": (ctypes.c_int, [_P, ctypes.c_int32, _P]),
    "minw_net_launches": (_I32, [_P]),
    "minw_net_kernels": (_I32, [_P]),
    "minw_net_destroy": (None, [_P]),
    "minw_get_last_device_error": (ctypes.c_int, [_P]),
}


def library_path():
    return _build.LIB


def lib(build_if_missing=False):
    """Load libminw.so.  Raises if it is missing: there is no other path."""
    global _LIB
    if _LIB is None:
        path = library_path()
        if not os.path.exists(path):
            if not build_if_missing:
                raise RuntimeError(f"libminw.so not built ({path}); run __graft_entry__.build()")
            _build.build()
        L = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _LIB = L
    return _LIB


def status_string(s):
    return lib().minw_status_string(int(s)).decode()


def _check(status, where):
    if status != MINW_OK:
        raise MinwError(status, where)


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("device tensor expected")
    if not t.is_contiguous():
        raise ValueError("contiguous tensor expected")
    return ctypes.c_void_p(t.data_ptr())


def _host_ptr(a):
    if isinstance(a, torch.Tensor):
        if a.is_cuda or not a.is_contiguous():
            raise ValueError("contiguous host tensor expected")
        return a.data_ptr()
    if not a.flags["C_CONTIGUOUS"]:
        raise ValueError("contiguous host array expected")
    return a.ctypes.data


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def quant(bits, thr=(0.0, 0.0, 0.0), scale=1.0):
    q = Quant()
    q.bits = int(bits)
    t = list(thr) + [0.0] * (3 - len(thr))
    for i in range(3):
        q.thr[i] = float(t[i])
    q.scale = float(scale)
    return q


def packed_words(N, C, H, W, bits):
    return N * H * W * bits * ((C + 31) // 32)


# ---------------------------------------------------------------------------
# entry points (same names as the C ABI)
# ---------------------------------------------------------------------------

def aqe_forward(x, y, alpha, q, stream=None):
    _check(lib().aqe_forward(_ptr(x), _ptr(y), x.numel(), float(alpha), ctypes.byref(q), _stream(stream)),
           "aqe_forward")


def aqe_forward_stochastic(x, y, alpha, seed, offset=0, stream=None):
    """Eq. our: alpha sign(x - z) + (1 - alpha) x, z ~ U[-1, 1) from
    Philox4x64-10 keyed by seed; offset advances the counter (ceil(n / 8) per
    call for fresh noise)."""
    _check(lib().aqe_forward_stochastic(_ptr(x), _ptr(y), x.numel(), float(alpha), int(seed) & (2**64 - 1),
                                        int(offset) & (2**64 - 1), _stream(stream)), "aqe_forward_stochastic")


def minw_to_bf16_nhwc(x, out, stream=None):
    """fp32 NCHW -> bf16 NHWC (out: a uint16 or bfloat16 tensor [B][H][W][C])."""
    B, C, H, W = x.shape
    _check(lib().minw_to_bf16_nhwc(_ptr(x), B, C, H, W, _ptr(out), _stream(stream)), "minw_to_bf16_nhwc")


def minw_pack_weight_bf16(w, q, out, channel_scale=None, stream=None):
    """Latent weights [O][C][kh][kw] -> bf16 level values [O][kh][kw][C]."""
    O, C, kh, kw = w.shape
    _check(lib().minw_pack_weight_bf16(_ptr(w), O, C, kh, kw, ctypes.byref(q), _ptr(channel_scale), _ptr(out),
                                       _stream(stream)), "minw_pack_weight_bf16")


def minw_to_bf16_nhwc_pad(x, Cp, out, stream=None):
    """fp32 NCHW -> bf16 NHWC with the channels padded to Cp (zeros) (out [B][H][W][Cp])."""
    B, C, H, W = x.shape
    _check(lib().minw_to_bf16_nhwc_pad(_ptr(x), B, C, H, W, int(Cp), _ptr(out), _stream(stream)),
           "minw_to_bf16_nhwc_pad")


def minw_pack_weight_bf16_pad(w, Cp, q, out, channel_scale=None, stream=None):
    """Latent weights [O][C][kh][kw] -> bf16 level values [O][kh][kw][Cp], channels past C zero."""
    O, C, kh, kw = w.shape
    _check(lib().minw_pack_weight_bf16_pad(_ptr(w), O, C, kh, kw, int(Cp), ctypes.byref(q), _ptr(channel_scale),
                                           _ptr(out), _stream(stream)), "minw_pack_weight_bf16_pad")


def minw_conv2d_bf16(act, B, C, H, W, wgt, O, kh, kw, bits_w, stride, pad, pool, scale, shift, y_out, stream=None):
    _check(lib().minw_conv2d_bf16(_ptr(act), B, C, H, W, _ptr(wgt), O, kh, kw, bits_w, stride, pad, int(pool),
                                  _ptr(scale), _ptr(shift), _ptr(y_out), _stream(stream)), "minw_conv2d_bf16")


def minw_conv2d_bf16_hardtanh(act, B, C, H, W, ldc, wgt, O, kh, kw, bits_w, stride, pad, scale, shift, out,
                              out_ld, out_off, residual=None, y_out=None, stream=None):
    _check(lib().minw_conv2d_bf16_hardtanh(_ptr(act), B, C, H, W, int(ldc), _ptr(wgt), O, kh, kw, bits_w, stride,
                                           pad, _ptr(scale), _ptr(shift), _ptr(out), int(out_ld), int(out_off),
                                           _ptr(residual), _ptr(y_out), _stream(stream)),
           "minw_conv2d_bf16_hardtanh")


def minw_bf16_matrix(x, out, transpose=False, stream=None):
    """fp32 matrix [rows][cols] -> bf16 (int16 bit patterns), transposed when asked,
    zero-padded to out's column count."""
    rows, cols = x.shape
    _check(lib().minw_bf16_matrix(_ptr(x), rows, cols, int(bool(transpose)), out.shape[1], _ptr(out),
                                  _stream(stream)), "minw_bf16_matrix")


def minw_sgd_clip(w, g, lr, stream=None):
    _check(lib().minw_sgd_clip(_ptr(w), _ptr(g), w.numel(), float(lr), _stream(stream)), "minw_sgd_clip")


def minw_fc_train_workspace_bytes(B, K, O):
    return int(lib().minw_fc_train_workspace_bytes(B, K, O))


def minw_fc_train_step(A, W, g_out, alpha, lr, q_w, q_a, a_out, g_in, workspace, a_pre=None, stream=None):
    """One Algorithm 1 step of a fully connected layer (W updated in place;
    a_pre, when given, receives the product before the activation AQE)."""
    B, K = A.shape
    O = W.shape[0]
    nbytes = workspace.numel() * workspace.element_size()
    _check(lib().minw_fc_train_step(_ptr(A), _ptr(W), _ptr(g_out), B, K, O, float(alpha), float(lr),
                                    ctypes.byref(q_w), ctypes.byref(q_a) if q_a is not None else None,
                                    _ptr(a_out), _ptr(g_in), _ptr(a_pre), _ptr(workspace), nbytes,
                                    _stream(stream)),
           "minw_fc_train_step")


def minw_conv_train_workspace_bytes(B, C, H, W, O, kh, kw, stride, pad):
    return int(lib().minw_conv_train_workspace_bytes(B, C, H, W, O, kh, kw, stride, pad))


def minw_conv_train_step(A, W, g_out, stride, pad, alpha, lr, q_w, q_a, a_out, g_in, workspace, a_pre=None,
                         stream=None):
    """One Algorithm 1 step of a convolutional layer: A [B][C][H][W], W
    [O][C][kh][kw] (updated in place), g_out [B][O][Ho][Wo]; a_pre, when
    given, receives the convolution before the activation AQE."""
    B, C, H, Wd = A.shape
    O, _, kh, kw = W.shape
    nbytes = workspace.numel() * workspace.element_size()
    _check(lib().minw_conv_train_step(_ptr(A), _ptr(W), _ptr(g_out), B, C, H, Wd, O, kh, kw, int(stride), int(pad),
                                      float(alpha), float(lr), ctypes.byref(q_w),
                                      ctypes.byref(q_a) if q_a is not None else None, _ptr(a_out), _ptr(g_in),
                                      _ptr(a_pre), _ptr(workspace), nbytes, _stream(stream)),
           "minw_conv_train_step")


def aqe_backward(x, gy, gx, alpha, stream=None):
    _check(lib().aqe_backward(_ptr(x), _ptr(gy), _ptr(gx), x.numel(), float(alpha), _stream(stream)),
           "aqe_backward")


def aqe_quantize_pack(x, q, planes, alpha=1.0, y=None, mask=None, stream=None):
    B, C, H, W = x.shape
    _check(lib().aqe_quantize_pack(_ptr(x), B, C, H, W, ctypes.byref(q), _ptr(planes), float(alpha),
                                   _ptr(y), _ptr(mask), _stream(stream)), "aqe_quantize_pack")


def aqe_backward_masked(mask, gy, gx, alpha, stream=None):
    _check(lib().aqe_backward_masked(_ptr(mask), _ptr(gy), _ptr(gx), gy.numel(), float(alpha),
                                     _stream(stream)), "aqe_backward_masked")


def minw_pack_weights(w, q, planes, channel_scale=None, stream=None):
    O, C, kh, kw = w.shape
    _check(lib().minw_pack_weights(_ptr(w), O, C, kh, kw, ctypes.byref(q), _ptr(channel_scale),
                                   _ptr(planes), _stream(stream)), "minw_pack_weights")


def minw_conv2d(act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad, acc_out=None,
                scale=None, shift=None, y_out=None, variant=VARIANT_AUTO, stream=None):
    _check(lib().minw_conv2d(_ptr(act), B, C, H, W, bits_a, _ptr(wgt), O, kh, kw, bits_w, stride, pad,
                             _ptr(acc_out), _ptr(scale), _ptr(shift), _ptr(y_out), int(variant),
                             _stream(stream)), "minw_conv2d")


def minw_conv_block(act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad, pool, scale, shift,
                    q_out=None, planes_out=None, y_out=None, variant=VARIANT_AUTO, stream=None):
    _check(lib().minw_conv_block(_ptr(act), B, C, H, W, bits_a, _ptr(wgt), O, kh, kw, bits_w, stride,
                                 pad, int(pool), _ptr(scale), _ptr(shift),
                                 ctypes.byref(q_out) if q_out is not None else None,
                                 _ptr(planes_out), _ptr(y_out), int(variant), _stream(stream)),
           "minw_conv_block")


def minw_conv_first(x, w, stride, pad, scale, shift, q_w=None, channel_scale=None, pool=0, q_out=None,
                    planes_out=None, y_out=None, stream=None):
    B, C, H, W = x.shape
    O, _, kh, kw = w.shape
    _check(lib().minw_conv_first(_ptr(x), B, C, H, W, _ptr(w), O, kh, kw, stride, pad,
                                 ctypes.byref(q_w) if q_w is not None else None, _ptr(channel_scale),
                                 int(pool), _ptr(scale), _ptr(shift),
                                 ctypes.byref(q_out) if q_out is not None else None,
                                 _ptr(planes_out), _ptr(y_out), _stream(stream)), "minw_conv_first")


def aqe_quantize_codes(x, q, codes, stream=None):
    B, C, H, W = x.shape
    _check(lib().aqe_quantize_codes(_ptr(x), B, C, H, W, ctypes.byref(q), _ptr(codes), _stream(stream)),
           "aqe_quantize_codes")


def minw_pack_weight_codes(w, q, codes, channel_scale=None, stream=None):
    O, C, kh, kw = w.shape
    _check(lib().minw_pack_weight_codes(_ptr(w), O, C, kh, kw, ctypes.byref(q), _ptr(channel_scale),
                                        _ptr(codes), _stream(stream)), "minw_pack_weight_codes")


def aqe_quantize_codes_e2m1(x, q, codes, stream=None):
    B, C, H, W = x.shape
    _check(lib().aqe_quantize_codes_e2m1(_ptr(x), B, C, H, W, ctypes.byref(q), _ptr(codes), _stream(stream)),
           "aqe_quantize_codes_e2m1")


def minw_pack_weight_codes_e2m1(w, q, codes, channel_scale=None, stream=None):
    O, C, kh, kw = w.shape
    _check(lib().minw_pack_weight_codes_e2m1(_ptr(w), O, C, kh, kw, ctypes.byref(q), _ptr(channel_scale),
                                             _ptr(codes), _stream(stream)), "minw_pack_weight_codes_e2m1")


def minw_conv2d_codes(act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad, acc_out=None,
                      scale=None, shift=None, y_out=None, stream=None):
    _check(lib().minw_conv2d_codes(_ptr(act), B, C, H, W, bits_a, _ptr(wgt), O, kh, kw, bits_w, stride, pad,
                                   _ptr(acc_out), _ptr(scale), _ptr(shift), _ptr(y_out), _stream(stream)),
           "minw_conv2d_codes")


def minw_conv_block_codes(act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad, pool, scale, shift,
                          q_out=None, codes_out=None, planes_out=None, y_out=None, stream=None):
    _check(lib().minw_conv_block_codes(_ptr(act), B, C, H, W, bits_a, _ptr(wgt), O, kh, kw, bits_w, stride,
                                       pad, int(pool), _ptr(scale), _ptr(shift),
                                       ctypes.byref(q_out) if q_out is not None else None,
                                       _ptr(codes_out), _ptr(planes_out), _ptr(y_out), _stream(stream)),
           "minw_conv_block_codes")


def minw_conv_block_codes_ex(act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad, pool, scale, shift,
                             q_out=None, codes_out=None, planes_out=None, y_out=None, res_codes=None, res_bits=0,
                             res_f32=None, y_nhwc=None, in_format=CODES_E4M3, out_format=CODES_E4M3,
                             res_format=CODES_E4M3, acc_out=None, e2m1_pairs=False, stream=None):
    ex = BlockExtra()
    ex.e2m1_pairs = int(bool(e2m1_pairs))
    ex.res_codes = res_codes.data_ptr() if res_codes is not None else None
    ex.res_bits = int(res_bits)
    ex.res_f32 = res_f32.data_ptr() if res_f32 is not None else None
    ex.y_nhwc = y_nhwc.data_ptr() if y_nhwc is not None else None
    ex.in_format, ex.out_format, ex.res_format = int(in_format), int(out_format), int(res_format)
    ex.acc_out = acc_out.data_ptr() if acc_out is not None else None
    _check(lib().minw_conv_block_codes_ex(_ptr(act), B, C, H, W, bits_a, _ptr(wgt), O, kh, kw, bits_w, stride, pad,
                                          int(pool), _ptr(scale), _ptr(shift),
                                          ctypes.byref(q_out) if q_out is not None else None, _ptr(codes_out),
                                          _ptr(planes_out), _ptr(y_out), ctypes.byref(ex), _stream(stream)),
           "minw_conv_block_codes_ex")


def minw_fc_workspace_bytes(B, K, O):
    return int(lib().minw_fc_workspace_bytes(B, K, O))


def minw_fc_ksplit(B, K, O, workspace_bytes):
    """K slices of minw_fc_codes for this shape and workspace size (host query)."""
    return lib().minw_fc_ksplit(int(B), int(K), int(O), int(workspace_bytes))


def minw_fc_codes(act, B, K, bits_a, wgt, O, bits_w, scale=None, shift=None, q_out=None, codes_out=None,
                  planes_out=None, y_out=None, acc_out=None, workspace=None, stream=None):
    nbytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().minw_fc_codes(_ptr(act), B, K, bits_a, _ptr(wgt), O, bits_w, _ptr(scale), _ptr(shift),
                               ctypes.byref(q_out) if q_out is not None else None, _ptr(codes_out),
                               _ptr(planes_out), _ptr(y_out), _ptr(acc_out), _ptr(workspace), nbytes,
                               _stream(stream)), "minw_fc_codes")


def minw_fc_codes_noalloc(act, B, K, bits_a, wgt, O, bits_w, scale=None, shift=None, q_out=None,
                          codes_out=None, planes_out=None, y_out=None, acc_out=None, stream=None):
    """minw_fc_codes with the library's fixed scratch array (allocates nothing)."""
    _check(lib().minw_fc_codes_noalloc(_ptr(act), B, K, bits_a, _ptr(wgt), O, bits_w, _ptr(scale), _ptr(shift),
                                       ctypes.byref(q_out) if q_out is not None else None, _ptr(codes_out),
                                       _ptr(planes_out), _ptr(y_out), _ptr(acc_out), _stream(stream)),
           "minw_fc_codes_noalloc")


def get_plan_options():
    o = PlanOptions()
    _check(lib().minw_get_plan_options(ctypes.byref(o)), "minw_get_plan_options")
    return {name: getattr(o, name) for name, _ in PlanOptions._fields_}


def set_plan_options(opts=None, **changes):
    """minw_set_plan_options: None and no changes restores the defaults;
    otherwise the current options (or opts) updated with changes."""
    if opts is None and not changes:
        _check(lib().minw_set_plan_options(None), "minw_set_plan_options")
        return
    cur = dict(opts if opts is not None else get_plan_options())
    cur.update(changes)
    o = PlanOptions(**cur)
    _check(lib().minw_set_plan_options(ctypes.byref(o)), "minw_set_plan_options")


def minw_measure_pipe_rates(stream=None):
    """minw_measure_pipe_rates as a dict (two-element lists for the N = 128 /
    N = 256 tensor-core rates)."""
    r = PipeRates()
    _check(lib().minw_measure_pipe_rates(ctypes.byref(r), _stream(stream)), "minw_measure_pipe_rates")
    out = {}
    for name, _ in PipeRates._fields_:
        v = getattr(r, name)
        out[name] = list(v) if hasattr(v, "__len__") else float(v)
    return out


def minw_test_stall_next_launch(kernel):
    _check(lib().minw_test_stall_next_launch(int(kernel)), "minw_test_stall_next_launch")


def minw_get_last_device_error(stream=None):
    return lib().minw_get_last_device_error(_stream(stream))


class Net:
    """Owner of a minw_net (minw_net_create / minw_forward / minw_net_destroy).

    ``layers`` is a list of dicts with the minw_layer_desc fields; ``w``,
    ``w_scale``, ``scale`` and ``shift`` are device tensors."""

    @classmethod
    def wresnet(cls, params, max_batch, device, stream=None, keep_activations=False):
        """minw_wresnet_create from a parameter dict shaped like
        ``inputs.wresnet_params`` (latent fp32 weights, BN maps); the tensors
        are copied to ``device`` for the call and released after it."""
        d = WResNetDesc()
        d.keep_activations = int(bool(keep_activations))
        d.n, d.bits_w = params["n"], params["bits_w"]
        for i in range(3):
            d.thr_w[i] = float(params["thr_w"][i])
        d.image_hw, d.num_classes = params["hw"], params["classes"]
        keep = []

        def dev(a):
            t = torch.from_numpy(a).to(device).contiguous()
            keep.append(t)
            return t.data_ptr()
        st = params["stem"]
        d.stem_w, d.stem_scale, d.stem_shift = dev(st["w"]), dev(st["scale"]), dev(st["shift"])
        nd = 0
        for b, blk in enumerate(params["blocks"]):
            c1, c2 = blk["c1"], blk["c2"]
            d.c1_w[b], d.c1_wscale[b], d.c1_scale[b], d.c1_shift[b] = (dev(c1["w"]), dev(c1["w_scale"]),
                                                                      dev(c1["scale"]), dev(c1["shift"]))
            d.c2_w[b], d.c2_wscale[b], d.c2_scale[b], d.c2_shift[b] = (dev(c2["w"]), dev(c2["w_scale"]),
                                                                      dev(c2["scale"]), dev(c2["shift"]))
            if blk["down"] is not None:
                c = blk["down"]
                d.down_w[nd], d.down_wscale[nd] = dev(c["w"]), dev(c["w_scale"])
                d.down_scale[nd], d.down_shift[nd] = dev(c["scale"]), dev(c["shift"])
                nd += 1
        fc = params["fc"]
        d.fc_w, d.fc_scale, d.fc_shift = dev(fc["w"]), dev(fc["scale"]), dev(fc["shift"])
        h = ctypes.c_void_p()
        _check(lib().minw_wresnet_create(ctypes.byref(d), int(max_batch), _stream(stream), ctypes.byref(h)),
               "minw_wresnet_create")
        net = cls.__new__(cls)
        net._h = h
        net.max_batch = max_batch
        net.out_features = params["classes"]
        return net

    def wresnet_activation(self, index, out, stream=None):
        """minw_wresnet_activation: the fp32 output of stage-step `index` of
        the most recent forward (0 the stem, b + 1 block b) into `out`."""
        _check(lib().minw_wresnet_activation(self._h, int(index), _ptr(out), out.numel(), _stream(stream)),
               "minw_wresnet_activation")

    @classmethod
    def wdense(cls, params, max_batch, device, stream=None):
        """minw_wdense_create from a parameter dict shaped like
        ``inputs.wdense_params`` (latent fp32 weights, BN maps); the tensors
        are copied to ``device`` for the call and released after it."""
        d = WDenseDesc()
        d.layers, d.growth, d.bits_w = params["layers"], params["growth"], params["bits_w"]
        for i in range(3):
            d.thr_w[i] = float(params["thr_w"][i])
        d.image_hw, d.num_classes = params["hw"], params["classes"]
        keep = []

        def dev(a):
            t = torch.from_numpy(a).to(device).contiguous()
            keep.append(t)
            return t.data_ptr()
        st = params["stem"]
        d.stem_w, d.stem_scale, d.stem_shift = dev(st["w"]), dev(st["scale"]), dev(st["shift"])
        j = 0
        for lay_list in params["blocks"]:
            for lay in lay_list:
                b, c = lay["b"], lay["c"]
                d.b_w[j], d.b_wscale[j], d.b_scale[j], d.b_shift[j] = (dev(b["w"]), dev(b["w_scale"]),
                                                                       dev(b["scale"]), dev(b["shift"]))
                d.c_w[j], d.c_wscale[j], d.c_scale[j], d.c_shift[j] = (dev(c["w"]), dev(c["w_scale"]),
                                                                       dev(c["scale"]), dev(c["shift"]))
                j += 1
        for i, t in enumerate(params["trans"]):
            d.t_w[i], d.t_wscale[i], d.t_scale[i], d.t_shift[i] = (dev(t["w"]), dev(t["w_scale"]),
                                                                   dev(t["scale"]), dev(t["shift"]))
        fc = params["fc"]
        d.fc_w, d.fc_scale, d.fc_shift = dev(fc["w"]), dev(fc["scale"]), dev(fc["shift"])
        h = ctypes.c_void_p()
        _check(lib().minw_wdense_create(ctypes.byref(d), int(max_batch), _stream(stream), ctypes.byref(h)),
               "minw_wdense_create")
        net = cls.__new__(cls)
        net._h = h
        net.max_batch = max_batch
        net.out_features = params["classes"]
        return net

    def wdense_features(self, block, out, stream=None):
        """minw_wdense_features: block `block`'s bf16 NHWC features after
        the most recent forward into the int16 device tensor `out`; returns
        (final channels, elements per pixel row)."""
        c, r = ctypes.c_int32(), ctypes.c_int32()
        _check(lib().minw_wdense_features(self._h, int(block), _ptr(out), out.numel(), ctypes.byref(c),
                                          ctypes.byref(r), _stream(stream)), "minw_wdense_features")
        return c.value, r.value

    @classmethod
    def resnet18(cls, params, max_batch, device, stream=None):
        """minw_resnet18_create from a parameter dict shaped like
        ``inputs.resnet18_params`` (latent fp32 weights, BN maps); the tensors
        are copied to ``device`` for the call and released after it."""
        d = ResNet18Desc()
        d.bits_a, d.bits_w = params["bits_a"], params["bits_w"]
        for i in range(3):
            d.thr_a[i] = float(params["thr_a"][i])
            d.thr_w[i] = float(params["thr_w"][i])
        d.image_hw, d.num_classes = params["hw"], params["classes"]
        keep = []

        def dev(a):
            t = torch.from_numpy(a).to(device).contiguous()
            keep.append(t)
            return t.data_ptr()
        st = params["stem"]
        d.stem_w, d.stem_scale, d.stem_shift = dev(st["w"]), dev(st["scale"]), dev(st["shift"])
        nd = 0
        for b, blk in enumerate(params["blocks"]):
            for j, c in enumerate((blk["c1"], blk["c2"])):
                d.conv_w[2 * b + j], d.conv_wscale[2 * b + j] = dev(c["w"]), dev(c["w_scale"])
                d.conv_scale[2 * b + j], d.conv_shift[2 * b + j] = dev(c["scale"]), dev(c["shift"])
            if blk["down"] is not None:
                c = blk["down"]
                d.down_w[nd], d.down_wscale[nd] = dev(c["w"]), dev(c["w_scale"])
                d.down_scale[nd], d.down_shift[nd] = dev(c["scale"]), dev(c["shift"])
                nd += 1
        fc = params["fc"]
        d.fc_w, d.fc_scale, d.fc_shift = dev(fc["w"]), dev(fc["scale"]), dev(fc["shift"])
        h = ctypes.c_void_p()
        _check(lib().minw_resnet18_create(ctypes.byref(d), int(max_batch), _stream(stream), ctypes.byref(h)),
               "minw_resnet18_create")
        net = cls.__new__(cls)
        net._h = h
        net.max_batch = max_batch
        net.out_features = params["classes"]
        return net

    def __init__(self, layers, max_batch, variant=VARIANT_AUTO, stream=None):
        arr = (LayerDesc * len(layers))()
        keep = []
        for d, L in zip(arr, layers):
            d.kind = L["kind"]
            d.C, d.H, d.W, d.O = L["C"], L["H"], L["W"], L["O"]
            d.kh, d.kw, d.stride, d.pad, d.pool = L.get("kh", 1), L.get("kw", 1), L.get("stride", 1), \
                L.get("pad", 0), int(L.get("pool", 0))
            d.bits_in, d.bits_w, d.bits_out = L["bits_in"], L["bits_w"], L["bits_out"]
            d.variant = int(L.get("variant", 0))
            for i in range(3):
                d.thr_w[i] = float(L["thr_w"][i])
                d.thr_out[i] = float(L["thr_out"][i])
            for k in ("w", "w_scale", "scale", "shift"):
                t = L.get(k)
                keep.append(t)
                setattr(d, k, t.data_ptr() if t is not None else None)
        h = ctypes.c_void_p()
        _check(lib().minw_net_create(arr, len(layers), int(max_batch), int(variant), _stream(stream),
                                     ctypes.byref(h)), "minw_net_create")
        self._h = h
        self.max_batch = max_batch
        self.out_features = layers[-1]["O"]

    def forward(self, x, logits, stream=None):
        _check(lib().minw_forward(self._h, _ptr(x), x.shape[0], _ptr(logits), _stream(stream)),
               "minw_forward")

    def forward_host(self, x_host, logits_host, stream=None):
        """Host-buffer forward (numpy or pinned CPU tensors): copies in, runs,
        copies the logits out and waits for them."""
        _check(lib().minw_forward_host(self._h, ctypes.c_void_p(_host_ptr(x_host)), x_host.shape[0],
                                       ctypes.c_void_p(_host_ptr(logits_host)), _stream(stream)),
               "minw_forward_host")

    def enable_timing(self, on=True):
        _check(lib().minw_net_enable_timing(self._h, int(on)), "minw_net_enable_timing")

    def layer_times(self):
        """Milliseconds of each layer's kernel in the most recent forward."""
        n = self.launches
        arr = (ctypes.c_float * n)()
        _check(lib().minw_net_layer_times(self._h, arr), "minw_net_layer_times")
        return list(arr)

    def layer_variants(self):
        """Kernel per layer: 0 fp32 first layer, VARIANT_POPC, VARIANT_TC (E4M3
        operands), VARIANT_TC_E2M1, VARIANT_TC_E2M1_PAIRS or VARIANT_TC_E2M1_N128."""
        n = self.launches
        arr = (ctypes.c_int32 * n)()
        _check(lib().minw_net_layer_variants(self._h, arr), "minw_net_layer_variants")
        return list(arr)

    def layer_candidates(self, layer):
        """Creation-time milliseconds of layer `layer`'s candidates under
        VARIANT_AUTO: [E4M3, E2M1, E2M1 pairs, popcount, E2M1 128-channel
        tiles], -1 where not one."""
        arr = (ctypes.c_float * 5)()
        _check(lib().minw_net_layer_candidates(self._h, int(layer), arr), "minw_net_layer_candidates")
        return list(arr)

    @property
    def kernels(self):
        """Kernels one forward launches."""
        return lib().minw_net_kernels(self._h)

    @property
    def launches(self):
        return lib().minw_net_launches(self._h)

    def close(self):
        if self._h:
            lib().minw_net_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def layer_descs(net_params, device):
    """minw_layer_desc dicts (device tensors) for a network described by
    ``inputs.convnet_params``: marshalling of the same fields, no compute."""
    out = []
    thr_a = net_params["thr_a"]
    c, h, w = net_params["in_shape"]
    for L in net_params["layers"]:
        d = dict(bits_in=L["bits_in"], bits_w=L["bits_w"], bits_out=L["bits_out"],
                 thr_w=list(net_params["thr_w"]), thr_out=list(thr_a) if L["bits_out"] else [0.0] * 3,
                 w=torch.from_numpy(L["w"]).to(device).contiguous(),
                 w_scale=torch.from_numpy(L["w_scale"]).to(device),
                 scale=torch.from_numpy(L["scale"]).to(device),
                 shift=torch.from_numpy(L["shift"]).to(device), O=L["O"])
        if L["kind"] == "conv":
            d.update(kind=LAYER_CONV, C=c, H=h, W=w, kh=L["kh"], kw=L["kw"], stride=L["stride"],
                     pad=L["pad"], pool=int(L["pool"]))
            h = (h + 2 * L["pad"] - L["kh"]) // L["stride"] + 1
            w = (w + 2 * L["pad"] - L["kw"]) // L["stride"] + 1
            if L["pool"]:
                h, w = h // 2, w // 2
            c = L["O"]
        else:
            d.update(kind=LAYER_FC, C=c, H=h, W=w)
            c, h, w = L["O"], 1, 1
        out.append(d)
    return out
