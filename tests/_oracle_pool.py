"""Oracle runs of the full-size parity tests spread over the host's cores.

The workers are spawned processes (never forked from a process that holds a
CUDA context); each rebuilds the seeded inputs of its task from the seeds,
so only seeds and indices cross the process boundary, and runs the CPU oracle
on them.  Test infrastructure only."""
import atexit
import functools
import multiprocessing as mp
import os

import numpy as np

_POOL = None


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def pool():
    global _POOL
    if _POOL is None:
        _POOL = mp.get_context("spawn").Pool(max(1, min(16, _cores())))
        atexit.register(_POOL.terminate)
    return _POOL


def starmap(fn, args):
    return pool().starmap(fn, list(args))


def spread(n, k=16):
    """k indices spread over range(n), first and last included."""
    return sorted(set(np.linspace(0, n - 1, min(k, n)).round().astype(int).tolist()))


@functools.lru_cache(maxsize=4)
def _convnet(seed, bits_a, bits_w, in_seed, batch):
    from paper_2003_04296_gb300.inputs import convnet_input, convnet_params
    return convnet_params(seed, bits_a=bits_a, bits_w=bits_w), convnet_input(in_seed, batch)


def convnet_logits(seed, bits_a, bits_w, in_seed, batch, i):
    """The oracle's logits of image i of the Model-A ConvNet workload."""
    from oracle import network as N
    p, x = _convnet(seed, bits_a, bits_w, in_seed, batch)
    return N.convnet_forward(p, x[i:i + 1])


@functools.lru_cache(maxsize=2)
def _resnet(seed, bits_a, bits_w, classes, hw, in_seed, batch):
    from paper_2003_04296_gb300.inputs import resnet18_input, resnet18_params
    return (resnet18_params(seed, bits_a=bits_a, bits_w=bits_w, classes=classes, hw=hw),
            resnet18_input(in_seed, batch, hw=hw))


def resnet_logits(seed, bits_a, bits_w, classes, hw, in_seed, batch, i):
    from oracle import network as N
    p, x = _resnet(seed, bits_a, bits_w, classes, hw, in_seed, batch)
    return N.resnet18_forward(p, x[i:i + 1])


@functools.lru_cache(maxsize=2)
def _conv(seed, B, C, H, W, O, k, stride, pad, x_dist, w_sigma):
    from paper_2003_04296_gb300.inputs import conv_problem
    return conv_problem(seed, B, C, H, W, O, k, k, stride, pad, 1, 1, x_dist=x_dist, w_sigma=w_sigma)


def conv_acc(spec, ba, bw, w_scale_kind, i):
    """Exact accumulators of image i of a standalone convolution problem
    (spec = the conv_problem arguments) at bit widths ba x bw; w_scale_kind
    'ones' or 'max' (1 / max |W[o]|)."""
    from oracle import oracle as O
    from paper_2003_04296_gb300.inputs import DEFAULT_THR
    p = _conv(*spec)
    ws = (np.ones(p["O"], np.float32) if w_scale_kind == "ones" else
          (1.0 / np.abs(p["w"].reshape(p["O"], -1)).max(1)).astype(np.float32))
    al = O.quantize(p["x"][i:i + 1], ba, DEFAULT_THR[ba])
    wl = O.quantize(p["w"], bw, DEFAULT_THR[bw], ws)
    return O.conv2d_levels(al, wl, p["stride"], p["pad"], ba, bw)
