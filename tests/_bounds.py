"""Error bounds of the GPU parity tests of the weight-only networks (numpy
and the oracle only): how far a tensor-core convolution with fp32
accumulation in its own summation order may land from the oracle's."""
import numpy as np

from oracle import oracle as O


def levels(conv, bits, thr):
    """A convolution's weight levels in integer units, as the oracle quantizes them."""
    return O.quantize(conv["w"], bits, thr, conv["w_scale"]) * 2.0 ** O.units_shift(bits)


def conv_bound(conv, xb, y_ref, stride, bits, thr, dx=None, channels=None):
    """Bound on |y_gpu - y_ref| of one weight-only convolution + BN whose
    bf16 input xb (fp64) is exact, or off by at most dx elementwise:
    |scale| K 2^-23 sum|x w| (fp32 accumulation in any order, rounding or
    truncating) + 2^-23 |y| (the BN fmaf), plus |scale| (dx conv |w|).
    K counts the channels the GPU sums over (``channels``: the zero-padded
    count, default xb's) times the taps."""
    k = conv["w"].shape[2]
    wl = np.abs(levels(conv, bits, thr))
    sc = np.abs(conv["scale"].astype(np.float64))[None, :, None, None]
    K = (channels or xb.shape[1]) * k * k
    mag = np.abs(xb) if dx is None else np.abs(xb) + dx
    A = O.conv2d_real(mag, wl, stride, k // 2)
    b = sc * K * 2.0 ** -23 * A + 2.0 ** -23 * np.abs(y_ref)
    if dx is not None:
        b = b + sc * O.conv2d_real(dx, wl, stride, k // 2)
    return b
