#!/usr/bin/env python3
"""Throughput of the MINW-Net inference path on GB300.

Default workload: the CIFAR-shaped Model-A ConvNet forward (conv 128-128-P-
256-256-P-512-512-P, FC 1024-1024-10), batch 256 per GPU, 1-bit activations x
1-bit weights in every hidden layer, fp32 image into the first layer, fp32
logits out.  ``--workload resnet18``: the ResNet-18-shaped network, batch 128
of 3x224x224 images, 3-bit activations and weights, fp32 stem and classifier.
Synthetic seeded data (images, latent weights, folded BN maps); no dataset.
One step = one minw_forward over the batch.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle on
a bounded sample of the same workload instead.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "MINW-Net conv effective binary TOPS and forward images/s; fraction of roofline"
L2_FLUSH_BYTES = 256 << 20
SMS = 152
SM_MAX_MHZ = 2070.0
POPC_PER_CLK_SM = 16          # measured: 16 popcounts per clock per SM
THROTTLE = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


def _measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["bf16_tflops"]), float(d.get("hbm_gbs", 6800.0))
    except (OSError, KeyError, ValueError):
        return 1900.0, 6800.0          # fallback figures of an earlier GB300 measurement


BF16_TFLOPS, HBM_GBS = _measured_peaks()

TRAFFIC_FILE = os.path.join(ROOT, "profiles", "conv_tc_cifar_convnet_a1w1_b256_traffic.json")


def _captured_traffic(bound):
    """DRAM bytes per launch of the tensor-core kernel from the committed ncu
    capture, or None when the kernel sources changed since the capture."""
    if bound != "tensor":
        return None
    try:
        import hashlib
        with open(TRAFFIC_FILE) as f:
            cap = json.load(f)
        h = hashlib.sha256()
        for src in cap["sources"]:
            with open(os.path.join(ROOT, src), "rb") as f:
                h.update(f.read())
        if h.hexdigest() != cap["sources_sha256"]:
            return None
        return cap["dram_bytes_per_launch"]
    except (OSError, KeyError, ValueError):
        return None
FP8_TFLOPS = 2.0 * BF16_TFLOPS        # nominal dense FP8 / bf16 = 4.5 / 2.25
FP4_TFLOPS = 6.0 * BF16_TFLOPS        # nominal dense FP4 / bf16 = 13.5 / 2.25
# tcgen05 rates this repository's pipe probe measured on GB300 (one CTA per SM,
# warp-uniform issue, M = 128, N = 256; bench.py --workload peaks re-measures them)
PROBE_TFLOPS = {"e4m3": 4826.0, "e2m1": 9673.0, "bf16": 2418.0}


def tensor_roofline(ops, kinds, ms):
    """Roofline of quantized layers on the tensor cores, each at the peak of its
    own operand kind ("e4m3" or "e2m1"): the time the layers would take at
    those peaks over the time they took.  Returns the roofline dict."""
    peak_of = {"e4m3": FP8_TFLOPS, "e2m1": FP4_TFLOPS}
    t_ms = sum(ms)
    t_roof = sum(o / (peak_of[k] * 1e12) for o, k in zip(ops, kinds)) * 1e3
    t_probe = sum(o / (PROBE_TFLOPS[k] * 1e12) for o, k in zip(ops, kinds)) * 1e3
    achieved = sum(ops) / (t_ms * 1e-3) / 1e12
    names = sorted(set(kinds))
    return {"bound": "tensor",
            "kernel": "conv_tc_kernel (tcgen05 " + " + ".join(
                {"e4m3": "kind::f8f6f4 E4M3", "e2m1": "kind::mxf4 E2M1"}[k] for k in names) + ")",
            "achieved": achieved, "peak": sum(ops) / (t_roof * 1e-3) / 1e12, "unit": "TFLOP/s",
            "frac": t_roof / t_ms, "traffic": None,
            "peak_basis": f"per layer: measured dense bf16 {BF16_TFLOPS:.1f} TFLOP/s (burst) x 2 for E4M3 and x 6 for "
                          "E2M1 layers (nominal FP8/FP4 to bf16 ratios), of measured",
            "peak_probe": sum(ops) / (t_probe * 1e-3) / 1e12,
            "frac_probe": t_probe / t_ms,
            "probe_basis": "per layer: the tcgen05 rate of its kind measured by this repository's pipe probe "
                           "(E4M3 4826, E2M1 9673 TFLOP/s at N = 256)",
            "layer_kinds": kinds}


L2_NOTE = "flushed between steps (256 MiB write outside the timed events)"


class Workload:
    """One benchmarked network: its seeded parameters and images, the net
    built through the library's API, the oracle forward, and the MACs of each
    op the net times (``minw_net_layer_times`` order)."""

    def __init__(self, name, args):
        from paper_2003_04296_gb300 import inputs as I
        self.name = name
        if name == "cifar_convnet":
            self.batch, self.seed = 256, 2
            self.model = getattr(args, "model", "A")
            self.params = I.convnet_params(self.seed, bits_a=args.bits_a, bits_w=args.bits_w,
                                           **I.CIFAR_MODELS[self.model])
            self.bits = (args.bits_a, args.bits_w)
        elif name == "wresnet110":
            self.batch, self.seed = 128, 6
            self.params = I.wresnet_params(self.seed, n=18, bits_w=3, classes=10, hw=32)
            self.bits = (0, 3)
        elif name == "wdense100":
            self.batch, self.seed = 128, 7
            self.params = I.wdense_params(self.seed, layers=16, growth=12, bits_w=3, classes=10, hw=32)
            self.bits = (0, 3)
        else:
            self.batch, self.seed = 128, 4
            self.params = I.resnet18_params(self.seed, bits_a=args.bits_a_resnet, bits_w=args.bits_w_resnet)
            self.bits = (args.bits_a_resnet, args.bits_w_resnet)

    def images(self, rank):
        from paper_2003_04296_gb300 import inputs as I
        if self.name == "cifar_convnet":
            return I.convnet_input(self.seed + 1000 * rank, self.batch)
        if self.name in ("wresnet110", "wdense100"):
            return I.wresnet_input(self.seed + 1000 * rank, self.batch)
        return I.resnet18_input(self.seed + 1000 * rank, self.batch)

    def net(self, minw, dev, variant, layer_variants=None):
        if self.name == "cifar_convnet":
            descs = minw.layer_descs(self.params, dev)
            if layer_variants:
                # a plan measured by an earlier run, replayed (e.g. under a profiler, whose
                # per-launch overhead would distort the creation-time measurement)
                for d, v in zip(descs, layer_variants):
                    d["variant"] = int(v)
            return minw.Net(descs, max_batch=self.batch, variant=variant)
        if self.name == "wresnet110":
            return minw.Net.wresnet(self.params, self.batch, dev)
        if self.name == "wdense100":
            return minw.Net.wdense(self.params, self.batch, dev)
        return minw.Net.resnet18(self.params, self.batch, dev)

    def oracle(self, x):
        from oracle import network as N
        if self.name == "cifar_convnet":
            return N.convnet_forward(self.params, x)
        if self.name == "wresnet110":
            return N.wresnet_forward(self.params, x)
        if self.name == "wdense100":
            return N.wdense_forward(self.params, x)
        return N.resnet18_forward(self.params, x)

    def op_macs(self):
        """MACs per image of each timed op, and the indices of the ops that
        run the quantized convolution (the roofline's kernel)."""
        if self.name == "cifar_convnet":
            m = layer_macs(self.params)
            return m, list(range(1, len(m)))
        if self.name == "wresnet110":
            # ops: stem, its pass; per block conv1, [shortcut], conv2 (HardTanh and the shortcut add fused); head
            # (unpadded MACs)
            hw = self.params["hw"]
            macs, q = [hw * hw * 16 * 27, 0], []
            size, c_in = hw, 16
            for blk in self.params["blocks"]:
                o = blk["c1"]["w"].shape[0]
                so = size // blk["stride"]
                q.append(len(macs)); macs.append(so * so * o * c_in * 9)
                if blk["down"] is not None:
                    q.append(len(macs)); macs.append(so * so * o * c_in)
                q.append(len(macs)); macs.append(so * so * o * o * 9)
                size, c_in = so, o
            macs.append(64 * self.params["classes"])
            return macs, q
        if self.name == "wdense100":
            # ops: stem, its pass; per layer 1x1, 3x3 (HardTanh fused in both); per transition conv, pool; head
            P = self.params
            hw, k = P["hw"], P["growth"]
            macs, q = [hw * hw * 2 * k * 27, 0], []
            for b, lay_list in enumerate(P["blocks"]):
                px = (hw >> b) ** 2
                for lay in lay_list:
                    c = lay["b"]["w"].shape[1]
                    q.append(len(macs)); macs.append(px * 4 * k * c)
                    q.append(len(macs)); macs.append(px * k * 4 * k * 9)
                if b < 2:
                    t = P["trans"][b]["w"]
                    q.append(len(macs)); macs += [px * t.shape[0] * t.shape[1], 0]
            macs.append(P["features"] * P["classes"])
            return macs, q
        hw = self.params["hw"]
        s = hw // 2
        macs = [s * s * 64 * 3 * 49, 0]
        size = s // 2
        for blk in self.params["blocks"]:
            o, c = blk["c1"]["w"].shape[:2]
            so = size // blk["stride"]
            macs.append(so * so * o * c * 9)
            if blk["down"] is not None:
                macs.append(so * so * o * c)
            macs.append(so * so * o * o * 9)
            size = so
        macs.append(512 * self.params["classes"])
        return macs, list(range(2, len(macs) - 1))

    def config(self, n_gpus):
        ba, bw = self.bits
        par = f"replicas x{n_gpus} (batch-sharded, no collective)"
        if self.name == "cifar_convnet":
            from paper_2003_04296_gb300.inputs import CIFAR_MODELS
            m = CIFAR_MODELS[self.model]
            w = m["widths"]
            layers = (f"conv3x3 {w[0]},{w[1]},P,{w[2]},{w[3]},P,{w[4]},{w[5]},P; "
                      f"fc {m['fcs'][0]},{m['fcs'][1]},10")
            tag = "" if self.model == "A" else f"_model{self.model}"
            return {"workload": f"cifar_convnet{tag}_fwd_a{ba}w{bw}", "batch_per_gpu": self.batch,
                    "global_batch": self.batch * n_gpus, "input": "3x32x32 fp32 U(-1,1)",
                    "layers": layers,
                    "bits_a": ba, "bits_w": bw, "first_layer": "fp32 input, quantized weights",
                    "parallelism": par, "l2": L2_NOTE}
        if self.name == "wresnet110":
            return {"workload": "wresnet110_cifar_fwd_w3", "batch_per_gpu": self.batch,
                    "global_batch": self.batch * n_gpus, "input": "3x32x32 fp32 U(-1,1)",
                    "layers": "stem 3x3 16 (fp32 weights); 3 x 18 basic blocks 16-32-64 (3-bit weights, bf16 "
                              "activations, 1x1/2 shortcuts entering stages 2-3); avgpool; fc 10 (fp32)",
                    "bits_a": "full precision (bf16 into each convolution)", "bits_w": bw,
                    "parallelism": par, "l2": L2_NOTE}
        if self.name == "wdense100":
            return {"workload": "densenet100_bc_k12_cifar_fwd_w3", "batch_per_gpu": self.batch,
                    "global_batch": self.batch * n_gpus, "input": "3x32x32 fp32 U(-1,1)",
                    "layers": "stem 3x3 24 (fp32 weights); 3 dense blocks x 16 bottleneck layers (1x1 to 48, 3x3 "
                              "to 12; 3-bit weights, bf16 activations) 24-216 / 108-300 / 150-342 channels; "
                              "transitions 1x1 + 2x2 avgpool (compression 1/2); avgpool; fc 10 (fp32)",
                    "bits_a": "full precision (bf16 into each convolution)", "bits_w": bw,
                    "parallelism": par, "l2": L2_NOTE}
        return {"workload": f"resnet18_fwd_a{ba}w{bw}", "batch_per_gpu": self.batch,
                "global_batch": self.batch * n_gpus, "input": "3x224x224 fp32 N(0,1)",
                "layers": "stem 7x7/2 64 + maxpool 3x3/2; basic blocks [2,2,2,2] 64-128-256-512; avgpool; fc 1000",
                "bits_a": ba, "bits_w": bw, "first_layer": "fp32 stem and classifier (fp32 weights)",
                "parallelism": par, "l2": L2_NOTE}


def max_over_ranks(v, world, device):
    """The largest v over the ranks (every rank gets it): the slowest replica
    sets the job's time."""
    import torch
    t = torch.tensor([float(v)], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_rank, world, seconds):
    """Whole-job throughput of independent replicas (weak scaling): every
    rank processes units_per_rank in `seconds` (the max over ranks)."""
    return units_per_rank * world / seconds


def layer_macs(net_p, hw=32):
    """MACs per image of each layer, in network order."""
    out = []
    size = hw
    for L in net_p["layers"]:
        if L["kind"] == "conv":
            out.append(size * size * L["O"] * L["C"] * L["kh"] * L["kw"])
            if L["pool"]:
                size //= 2
        else:
            out.append(L["O"] * L["K"])
    return out


# ------------------------------------------------------------------ clocks --

class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during timing."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
            # the timed region starts once the sampler is running (first line written)
            t0 = time.time()
            while time.time() - t0 < 5.0 and os.path.getsize(self.path) == 0 and self.proc.poll() is None:
                time.sleep(0.02)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.out.close()

    def summary(self):
        if self.proc is None or not self.path:
            return None
        mhz, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    mhz.append(float(parts[1]))
                    mx = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not mhz:
            return None
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(mhz)}


# --------------------------------------------------------------- reference --

def oracle_images_per_s(wl, x, max_seconds):
    """Time the oracle's network forward image by image until max_seconds."""
    wl.oracle(x[:1])                          # builds and loads the oracle
    done, t0 = 0, time.perf_counter()
    while done < x.shape[0]:
        wl.oracle(x[done:done + 1])
        done += 1
        if time.perf_counter() - t0 >= max_seconds:
            break
    dt = time.perf_counter() - t0
    return done / dt, done, dt


def _oracle_worker(job):
    """One process of the all-cores oracle baseline: the network forward of
    its images, one by one, until its time is up (returns images done, s)."""
    name, bits, lo, n, seconds = job
    import argparse as _ap
    a = _ap.Namespace(bits_a=bits[0], bits_w=bits[1], model="A", bits_a_resnet=bits[0], bits_w_resnet=bits[1])
    wl = Workload(name, a)
    x = wl.images(0)[lo:lo + n]
    wl.oracle(x[:1])
    done, t0 = 0, time.perf_counter()
    while done < x.shape[0] and time.perf_counter() - t0 < seconds:
        wl.oracle(x[done:done + 1])
        done += 1
    return done, time.perf_counter() - t0


def oracle_all_cores(name, bits, batch, seconds):
    """The oracle forward on every core of this process's affinity mask, as
    independent processes (spawned: no state shared with the GPU context),
    each over its own images of the batch: aggregate images/s."""
    import multiprocessing as mp
    try:
        cores = len(os.sched_getaffinity(0))
    except AttributeError:
        cores = os.cpu_count() or 1
    per = max(1, batch // cores)
    jobs = [(name, bits, (i * per) % batch, per, seconds) for i in range(cores)]
    ctx = mp.get_context("spawn")
    with ctx.Pool(cores) as pool:
        res = pool.map(_oracle_worker, jobs)
    imgs = sum(r[0] for r in res)
    span = max(r[1] for r in res)
    return imgs / span, imgs, span, cores


def cpu_model():
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu model")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def run_reference_conv1(args):
    """The oracle on the single convolution: whole steps (quantize, fp64
    level convolution, BN) of the 4-image batch."""
    from oracle import oracle as Or
    from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem
    p = conv_problem(0, 4, 128, 32, 32, 128, 3, 3, 1, 1, 1, 1)
    mac = 4 * 32 * 32 * 128 * 128 * 9
    times = []
    for k in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        al = Or.quantize(p["x"], 1, DEFAULT_THR[1])
        wl = Or.quantize(p["w"], 1, DEFAULT_THR[1], p["w_scale"])
        Or.affine(Or.conv2d_levels(al, wl, 1, 1, 1, 1), p["scale"], p["shift"])
        if k >= args.warmup:
            times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    tops = 2.0 * mac / sec / 1e12
    line = {"metric": METRIC, "value": tops, "unit": "effective TOPS (2 x MAC / s)", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
            "impl": "reference", "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": conv1_config(args.gpus),
            "cpu_baseline": {"value": tops, "unit": "effective TOPS", "cores": 1, "kind": "oracle",
                             "sample": "whole steps of the 4-image workload, single-threaded C oracle"},
            "e2e": {"value": tops, "unit": "effective TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_reference_sweep(args):
    """The oracle on the sweep: one image per step through the fp64 level
    convolution, cycling through the nine bit-width pairs."""
    from oracle import oracle as Or
    from paper_2003_04296_gb300.inputs import DEFAULT_THR
    p = sweep_problem()
    mac_img = 14 * 14 * 512 * 512 * 9
    times = []
    for k in range(args.warmup + args.steps):
        ba, bw = SWEEP_PAIRS[k % len(SWEEP_PAIRS)]
        a_lv = Or.quantize(p["x"][k % 256:k % 256 + 1], ba, DEFAULT_THR[ba])
        w_lv = Or.quantize(p["w"], bw, DEFAULT_THR[bw], p["w_scale"])
        t0 = time.perf_counter()
        Or.conv2d_levels(a_lv, w_lv, 1, 1, ba, bw)
        if k >= args.warmup:
            times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    tops = 2.0 * mac_img / sec / 1e12
    sample = "one image per step (of 256) through the fp64 oracle convolution, the nine pairs in turn"
    line = {"metric": METRIC, "value": tops, "unit": "effective TOPS (2 x MAC / s)", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
            "impl": "reference", "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": sweep_config(args.gpus),
            "cpu_baseline": {"value": tops, "unit": "effective TOPS", "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": tops, "unit": "effective TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_reference(args, rank):
    if rank != 0:
        return None
    if args.workload == "sweep":
        return run_reference_sweep(args)
    if args.workload == "fc_train":
        return run_reference_fc_train(args)
    if args.workload == "conv_train":
        return run_reference_conv_train(args)
    if args.workload == "conv1":
        return run_reference_conv1(args)
    wl = Workload(args.workload, args)
    x = wl.images(0)
    B = wl.batch
    # per-step sample sized so that warmup + steps stay within ~3 minutes
    t0 = time.perf_counter()
    wl.oracle(x[:1])
    t_img = time.perf_counter() - t0
    per_step = max(1, min(B, int(150.0 / max(args.warmup + args.steps, 1) / max(t_img, 1e-3))))
    for _ in range(args.warmup):
        wl.oracle(x[:per_step])
    times = []
    for k in range(args.steps):
        lo = (k * per_step) % B
        xs = x[lo:lo + per_step]
        t0 = time.perf_counter()
        wl.oracle(xs)
        times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    ips = per_step / sec
    sample = f"{per_step} of the {B} images per step, single-threaded C oracle, extrapolated to images/s"
    line = {"metric": METRIC, "value": ips, "unit": "images/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True, "impl": "reference",
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": wl.config(args.gpus),
            "cpu_baseline": {"value": ips, "unit": "images/s", "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": ips, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------- GPU --

def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    import __graft_entry__ as g
    if rank == 0:
        g.build()
    if world > 1:
        dist.barrier()
    from paper_2003_04296_gb300 import minw

    wl = Workload(args.workload, args)
    BATCH = wl.batch
    x_np = wl.images(rank)
    lv = [int(v) for v in args.layer_variants.split(",")] if getattr(args, "layer_variants", None) else None
    net = wl.net(minw, dev, args.variant, lv)
    x = torch.from_numpy(x_np).to(dev)
    logits = torch.empty((BATCH, net.out_features), dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    macs, q_ops_idx = wl.op_macs()
    nl = net.launches
    assert len(macs) == nl, (len(macs), nl)

    for _ in range(max(args.warmup, 3)):
        net.forward(x, logits)
    torch.cuda.synchronize()

    step_ms, layer_ms = [], np.zeros(nl)
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clk:
        for k in range(args.steps):
            flush.zero_()                       # evict the previous step from L2
            ev0[k].record(stream)
            net.forward(x, logits)
            ev1[k].record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
    # per-kernel durations: the same K steps again with an event after every
    # layer (events between kernels stop a kernel's set-up from overlapping the
    # previous one's tail, so the timed steps above run without them)
    net.enable_timing(True)
    for k in range(args.steps):
        flush.zero_()
        net.forward(x, logits)
        layer_ms += np.array(net.layer_times())
    net.enable_timing(False)
    torch.cuda.synchronize()
    for k in range(args.steps):
        step_ms.append(ev0[k].elapsed_time(ev1[k]))
    ms_max = max_over_ranks(sum(step_ms) / len(step_ms), world, dev)

    # end to end through the public API: pinned host input -> logits on host
    x_host = torch.from_numpy(x_np).pin_memory()
    out_host = torch.empty((BATCH, net.out_features), dtype=torch.float32).pin_memory()
    net.enable_timing(False)
    for _ in range(2):
        net.forward_host(x_host, out_host)
    e2e_s = []
    if world > 1:
        dist.barrier()
    for _ in range(args.steps):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        net.forward_host(x_host, out_host)
        e2e_s.append(time.perf_counter() - t0)
    e2e_sec = max_over_ranks(sum(e2e_s) / len(e2e_s), world, dev)

    if rank != 0:
        return None

    clocks = clk.summary()
    layer_ms /= args.steps
    total_macs = sum(macs) * BATCH
    value = replica_throughput(BATCH, world, ms_max * 1e-3)
    eff_tops = replica_throughput(2.0 * total_macs, world, ms_max * 1e-3) / 1e12

    # roofline of the dominant kernel: the quantized convolution (every op in q_ops_idx)
    variants = net.layer_variants()
    q_ms = float(sum(layer_ms[i] for i in q_ops_idx))
    q_ops = 2.0 * sum(macs[i] for i in q_ops_idx) * BATCH
    achieved = q_ops / (q_ms * 1e-3) / 1e12
    tc_kind = {minw.VARIANT_TC: "e4m3", minw.VARIANT_TC_E2M1: "e2m1", minw.VARIANT_TC_E2M1_PAIRS: "e2m1",
               minw.VARIANT_TC_E2M1_N128: "e2m1"}
    if wl.name in ("wresnet110", "wdense100"):
        tc_kind = {minw.VARIANT_TC: "bf16"}
    all_tc = all(variants[i] in tc_kind for i in q_ops_idx)
    if wl.name == "wresnet110":
        roofline = {"bound": "tensor", "kernel": "conv_tc_kernel<0, *, bf16> (tcgen05 kind::f16, the 110 block "
                                                 "and shortcut convolutions)",
                    "achieved": achieved, "peak": BF16_TFLOPS, "unit": "TFLOP/s", "frac": achieved / BF16_TFLOPS,
                    "traffic": None, "layer_kinds": ["bf16"] * len(q_ops_idx),
                    "peak_basis": "measured dense bf16 TFLOP/s (burst), of measured; achieved counts the unpadded "
                                  "MACs (16- and 32-channel layers run on operands padded to 64 channels)"}
    elif wl.name == "wdense100":
        roofline = {"bound": "tensor", "kernel": "conv_tc_kernel<0, *, bf16> (tcgen05 kind::f16, the 96 "
                                                 "bottleneck-layer and 2 transition convolutions)",
                    "achieved": achieved, "peak": BF16_TFLOPS, "unit": "TFLOP/s", "frac": achieved / BF16_TFLOPS,
                    "traffic": None, "layer_kinds": ["bf16"] * len(q_ops_idx),
                    "peak_basis": "measured dense bf16 TFLOP/s (burst), of measured; achieved counts the unpadded "
                                  "MACs (each 1x1 reads its channels padded to a multiple of 64, the 3x3 its 48 "
                                  "padded to 64, and the 3x3 computes 12 output channels of a 16-wide MMA)"}
    elif all_tc:
        roofline = tensor_roofline([2.0 * macs[i] * BATCH for i in q_ops_idx],
                                   [tc_kind[variants[i]] for i in q_ops_idx],
                                   [float(layer_ms[i]) for i in q_ops_idx])
    else:
        peak = POPC_PER_CLK_SM * 32 * 2 * SMS * SM_MAX_MHZ * 1e6 / 1e12
        roofline = {"bound": "alu", "kernel": "conv_popc_kernel (all quantized layers)",
                    "achieved": achieved, "peak": peak, "unit": "TOPS (2 x binary MAC)",
                    "frac": achieved / peak, "traffic": None,
                    "peak_basis": "16 popc/clk/SM x 32 MAC/popc x 2 ops x 152 SMs x 2070 MHz"}
    roofline["layer_variants"] = variants
    roofline["traffic"] = _captured_traffic(roofline["bound"]) if wl.name == "cifar_convnet" else None

    cpu = cpu_all = None
    if world == 1 and not args.skip_cpu:
        ips, n_img, secs = oracle_images_per_s(wl, x_np, args.cpu_seconds)
        cpu = {"value": ips, "unit": "images/s", "cores": 1, "kind": "oracle",
               "sample": f"{n_img} images of the batch through the single-threaded C oracle ({secs:.1f} s)",
               "cpu": cpu_model()}
        ips_all, n_all, secs_all, cores = oracle_all_cores(wl.name, wl.bits, BATCH, args.cpu_seconds)
        cpu_all = {"value": ips_all, "unit": "images/s", "cores": cores, "kind": "oracle",
                   "sample": f"{n_all} images through {cores} independent single-threaded oracle processes "
                             f"(one per core of the affinity mask, spawned), {secs_all:.1f} s",
                   "cpu": cpu_model()}

    line = {"metric": METRIC, "value": value, "unit": "images/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None,
            "dtype": ("+".join(sorted(set(roofline["layer_kinds"]))) if all_tc else "b1"),
            "data": "synthetic",
            "config": wl.config(world),
            "eff_tops": eff_tops,
            "layer_ms": [round(v, 5) for v in layer_ms.tolist()],
            "layer_ms_note": "per-op CUDA-event durations from a second pass of the same steps with an event "
                             "after every op; the timed steps run without them",
            "roofline": roofline, "cpu_baseline": cpu, "cpu_baseline_all_cores": cpu_all,
            "e2e": {"value": replica_throughput(BATCH, world, e2e_sec), "unit": "images/s",
                    "h2d_bytes_per_step": int(x_host.numel() * 4),
                    "d2h_bytes_per_step": int(out_host.numel() * 4)},
            "gpu_launches": net.kernels * args.steps, "clocks": clocks}
    return line


# ------------------------------------------------------------------ sweep --

SWEEP_PAIRS = [(a, w) for a in (1, 2, 3) for w in (1, 2, 3)]


def sweep_problem():
    from paper_2003_04296_gb300.inputs import conv_problem
    return conv_problem(5, 256, 512, 14, 14, 512, 3, 3, 1, 1, 1, 1, x_dist="normal", w_sigma=1.0)


def sweep_config(n_gpus):
    return {"workload": "conv3x3_bitwidth_sweep_256x512x14x14_to512", "batch_per_gpu": 256,
            "global_batch": 256 * n_gpus, "input": "256x512x14x14 fp32 N(0,1), weights 512x512x3x3 N(0,1)",
            "pairs": "(bits_a, bits_w) in {1,2,3}^2, each a 3x3/1/1 convolution to int32 accumulators",
            "aqe": "AQE forward (alpha 0.75) and backward on the same 25.7M-element tensor (the stochastic forward, "
                   "Eq. our, is timed beside the steps)",
            "parallelism": f"replicas x{n_gpus} (batch-sharded, no collective)", "l2": L2_NOTE}


# ------------------------------------------------------------ single conv --

def conv1_config(n_gpus):
    return {"workload": "conv3x3_4x128x32x32_to128_a1w1", "batch_per_gpu": 4, "global_batch": 4 * n_gpus,
            "input": "4x128x32x32 fp32 N(0,1), weights 128x128x3x3 N(0,0.05), seed 0",
            "step": "quantize the input to E2M1 codes (Eq. inference, 1-bit), then the 3x3/1/1 convolution "
                    "with int32 accumulators and the fp32 per-channel BN output; weights packed once",
            "launch": "each timed step replays a CUDA graph of the step's two kernels",
            "parallelism": f"replicas x{n_gpus} (batch-sharded, no collective)", "l2": L2_NOTE}


def run_conv1(args, rank, world, local_rank):
    """The single quantized convolution of the smallest workload: the step
    quantizes the fp32 input and convolves it (int32 accumulators plus the
    fp32 BN output).  The op is a few microseconds, so each step replays a
    CUDA graph of the two launches (the L2 flush stays outside the graph)."""
    import torch
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    import __graft_entry__ as g
    if rank == 0:
        g.build()
    from paper_2003_04296_gb300 import minw
    from paper_2003_04296_gb300.inputs import DEFAULT_THR, conv_problem
    B, C, H, W, O = 4, 128, 32, 32, 128
    p = conv_problem(0, B, C, H, W, O, 3, 3, 1, 1, 1, 1)
    x = torch.from_numpy(p["x"]).to(dev)
    sc, sh = torch.from_numpy(p["scale"]).to(dev), torch.from_numpy(p["shift"]).to(dev)
    act = torch.empty((B, H, W, C // 2), dtype=torch.uint8, device=dev)
    wgt = torch.empty((O, 3, 3, C // 2), dtype=torch.uint8, device=dev)
    minw.minw_pack_weight_codes_e2m1(torch.from_numpy(p["w"]).to(dev), minw.quant(1, DEFAULT_THR[1]), wgt,
                                     channel_scale=torch.from_numpy(p["w_scale"]).to(dev))
    acc = torch.empty((B, O, H, W), dtype=torch.int32, device=dev)
    y = torch.empty((B, O, H, W), dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    s = torch.cuda.Stream(device=dev)
    q = minw.quant(1, DEFAULT_THR[1])

    def step(stream):
        minw.aqe_quantize_codes_e2m1(x, q, act, stream=stream)
        minw.minw_conv_block_codes_ex(act, B, C, H, W, 1, wgt, O, 3, 3, 1, 1, 1, 0, sc, sh, y_out=y,
                                      in_format=minw.CODES_E2M1, acc_out=acc, stream=stream)

    with torch.cuda.stream(s):
        for _ in range(3):
            step(s)
    s.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        step(torch.cuda.current_stream())
    torch.cuda.synchronize()
    for _ in range(max(args.warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    cur = torch.cuda.current_stream()
    with ClockSampler(local_rank) as clk:
        for k in range(args.steps):
            flush.zero_()
            e0[k].record(cur)
            graph.replay()
            e1[k].record(cur)
        torch.cuda.synchronize()
    ms = sum(e0[k].elapsed_time(e1[k]) for k in range(args.steps)) / args.steps
    ms_max = max_over_ranks(ms, world, dev)
    # per-kernel time of the convolution (direct launches with events around it)
    cms = []
    for k in range(min(args.steps, 200)):
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        flush.zero_()
        minw.aqe_quantize_codes_e2m1(x, q, act)
        a0.record(cur)
        minw.minw_conv_block_codes_ex(act, B, C, H, W, 1, wgt, O, 3, 3, 1, 1, 1, 0, sc, sh, y_out=y,
                                      in_format=minw.CODES_E2M1, acc_out=acc)
        a1.record(cur)
        torch.cuda.synchronize()
        cms.append(a0.elapsed_time(a1))
    conv_ms = float(np.median(cms))
    # end to end: pinned host input in, accumulators and BN output back
    x_host = torch.from_numpy(p["x"]).pin_memory()
    acc_host = torch.empty(acc.shape, dtype=torch.int32).pin_memory()
    y_host = torch.empty(y.shape, dtype=torch.float32).pin_memory()
    e2e_s = []
    for k in range(min(args.steps, 200) + 1):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        x.copy_(x_host, non_blocking=True)
        graph.replay()
        acc_host.copy_(acc, non_blocking=True)
        y_host.copy_(y, non_blocking=True)
        torch.cuda.synchronize()
        if k:
            e2e_s.append(time.perf_counter() - t0)
    e2e_sec = max_over_ranks(sum(e2e_s) / len(e2e_s), world, dev)
    if rank != 0:
        return None
    mac = B * H * W * O * C * 9
    roofline = tensor_roofline([2.0 * mac], ["e2m1"], [conv_ms])
    roofline["kernel"] = "conv_tc_kernel (tcgen05 kind::mxf4 E2M1; int32 and fp32 NCHW outputs)"
    roofline["note"] = ("a 6.0e8-MAC layer: one wave of 32 tiles with 9 K blocks each, so launch and "
                        "pipeline fill set its time, not the tensor pipe")
    cpu = None
    if world == 1 and not args.skip_cpu:
        from oracle import oracle as Or
        t0, n = time.perf_counter(), 0
        while True:
            al = Or.quantize(p["x"], 1, DEFAULT_THR[1])
            wl = Or.quantize(p["w"], 1, DEFAULT_THR[1], p["w_scale"])
            Or.affine(Or.conv2d_levels(al, wl, 1, 1, 1, 1), p["scale"], p["shift"])
            n += 1
            if time.perf_counter() - t0 > min(args.cpu_seconds, 10.0):
                break
        dt = time.perf_counter() - t0
        cpu = {"value": 2.0 * mac * n / dt / 1e12, "unit": "effective TOPS", "cores": 1, "kind": "oracle",
               "sample": f"{n} whole steps of the workload (quantize, fp64 level convolution, BN) in {dt:.1f} s"}
    return {"metric": METRIC, "value": replica_throughput(2.0 * mac, world, ms_max * 1e-3) / 1e12,
            "unit": "effective TOPS (2 x MAC / s)", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "e2m1", "data": "synthetic", "config": conv1_config(world), "conv_ms": round(conv_ms, 5),
            "roofline": roofline, "cpu_baseline": cpu,
            "e2e": {"value": 2.0 * mac * world / e2e_sec / 1e12, "unit": "effective TOPS",
                    "h2d_bytes_per_step": int(x_host.numel() * 4),
                    "d2h_bytes_per_step": int(acc_host.numel() * 4 + y_host.numel() * 4)},
            "gpu_launches": 2 * args.steps, "clocks": clk.summary()}


def step_bytes(B, K, O):
    """Bytes one fully connected training step moves at least, launch by launch:
    the weight pass (W read, its bf16 copy and transposed copy written), the
    activation pass (a read, two bf16 copies written), the forward product
    (bf16 a and W^ read, a~ written), the gradient pass (a~ and g read, a_out
    and two bf16 copies of g~ written), the input-gradient product (bf16 g~
    and W^T read, g_in written) and the weight-gradient product with the
    update (bf16 g~^T and a^T read, W read and written)."""
    Op = (O + 63) // 64 * 64
    OK, BK, BO = O * K, B * K, B * O
    return float(6 * OK + 2 * K * Op + 8 * BK + (2 * BK + 2 * OK + 4 * BO) + (12 * BO + 2 * B * Op + 2 * O * B)
                 + (2 * B * Op + 2 * K * Op + 4 * BK) + (2 * O * B + 2 * K * B + 8 * OK))


FC_TRAIN_SHAPE = (256, 8192, 1024)       # batch, K, O: fc1 of the CIFAR model
FC_TRAIN_ALPHA, FC_TRAIN_LR = 0.75, 1e-3


def fc_train_problem(rank=0):
    """Seeded input, latent weights and upstream gradient of the training
    workload (fp32 numpy)."""
    B, K, O = FC_TRAIN_SHAPE
    r = np.random.default_rng(31 + 1000 * rank)
    A = np.clip(r.standard_normal((B, K)), -1.5, 1.5).astype(np.float32)
    W = r.uniform(-1, 1, (O, K)).astype(np.float32)
    G = (r.standard_normal((B, O)) * 0.1).astype(np.float32)
    return A, W, G


def fc_train_oracle_rate(A, W, G, budget_s=10.0, warmup=1, max_steps=30):
    """The oracle's training step (oracle.fc_train_step), timed on the host:
    whole steps until budget_s seconds; returns (images/s, s per step, steps)."""
    from oracle import oracle as Or
    from paper_2003_04296_gb300.inputs import DEFAULT_THR
    qw, qa = (1, DEFAULT_THR[1]), (1, DEFAULT_THR[1])
    for _ in range(warmup):
        Or.fc_train_step(A, W, G, FC_TRAIN_ALPHA, FC_TRAIN_LR, qw[0], qw[1], qa)
    times = []
    t_start = time.perf_counter()
    while len(times) < max_steps and (not times or time.perf_counter() - t_start < budget_s):
        t0 = time.perf_counter()
        Or.fc_train_step(A, W, G, FC_TRAIN_ALPHA, FC_TRAIN_LR, qw[0], qw[1], qa)
        times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    return A.shape[0] / sec, sec, len(times)


def fc_train_config(world):
    B, K, O = FC_TRAIN_SHAPE
    return {"workload": "fc_train_8192x1024_b256_a1w1", "batch_per_gpu": B, "global_batch": B * world,
            "layer": f"FC {K} -> {O} (Model A's fc1), alpha {FC_TRAIN_ALPHA}, lr {FC_TRAIN_LR}, SGD + clip",
            "parallelism": f"replicas x{world} (no gradient all-reduce)", "l2": L2_NOTE}


def run_reference_fc_train(args):
    """The oracle's training step on the training workload, whole steps."""
    A, W, G = fc_train_problem(0)
    ips, sec, n = fc_train_oracle_rate(A, W, G, budget_s=1e9, warmup=args.warmup, max_steps=args.steps)
    sample = (f"{n} full steps of the batch through oracle.fc_train_step (numpy's BLAS threads for the three fp64 "
              "products, single-threaded C for the elementwise stages)")
    line = {"metric": "Algorithm 1 training step of a fully connected MINW layer: images/s", "value": ips,
            "unit": "images/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": sec * 1e3, "higher_is_better": True, "impl": "reference", "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": fc_train_config(args.gpus),
            "cpu_baseline": {"value": ips, "unit": "images/s", "cores": os.cpu_count(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": ips, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_fc_train(args, rank, world, local_rank):
    """Algorithm 1's training step of Model A's first fully connected layer
    (8192 -> 1024, batch 256, 1-bit weights and activations, alpha 0.75): the
    weight AQE, the forward product, the activation AQE and its backward mask,
    the input and weight gradients, the mask of Eq. weight and the clipped
    update, through minw_fc_train_step.  Its three tensor-core products hold
    6 B K O flops over about 200 MB of operands and results: the step is bound
    by HBM, and its roofline counts the bytes each of its launches must move
    at least (step_bytes), over the step's event time."""
    import torch
    import __graft_entry__ as g
    if rank == 0:
        g.build()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    from paper_2003_04296_gb300 import minw
    from paper_2003_04296_gb300.inputs import DEFAULT_THR
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    B, K, O = FC_TRAIN_SHAPE
    A_np, W_np, G_np = fc_train_problem(rank)
    A, W, G = (torch.from_numpy(x).to(dev) for x in (A_np, W_np, G_np))
    a_out = torch.empty((B, O), device=dev)
    g_in = torch.empty((B, K), device=dev)
    ws = torch.empty(minw.minw_fc_train_workspace_bytes(B, K, O), dtype=torch.uint8, device=dev)
    qw, qa = minw.quant(1, DEFAULT_THR[1]), minw.quant(1, DEFAULT_THR[1])
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        minw.minw_fc_train_step(A, W, G, FC_TRAIN_ALPHA, FC_TRAIN_LR, qw, qa, a_out, g_in, ws)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    with ClockSampler(local_rank) as clk:
        for k in range(args.steps):
            flush.zero_()
            e0[k].record(stream)
            step()
            e1[k].record(stream)
        torch.cuda.synchronize()
    ms_max = max_over_ranks(sum(e0[k].elapsed_time(e1[k]) for k in range(args.steps)) / args.steps, world, dev)
    # end to end: the batch and the upstream gradient from pinned host memory, the input gradient back
    A_host = A.cpu().pin_memory()
    G_host = G.cpu().pin_memory()
    gin_host = torch.empty((B, K), dtype=torch.float32).pin_memory()
    e2e_s = []
    for k in range(min(args.steps, 20) + 1):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        A.copy_(A_host, non_blocking=True)
        G.copy_(G_host, non_blocking=True)
        step()
        gin_host.copy_(g_in, non_blocking=True)
        torch.cuda.synchronize()
        if k:
            e2e_s.append(time.perf_counter() - t0)
    e2e_sec = max_over_ranks(sum(e2e_s) / len(e2e_s), world, dev)
    if rank != 0:
        return None
    cpu = None
    if world == 1 and not args.skip_cpu:
        ips, sec, n = fc_train_oracle_rate(A_np, W_np, G_np, budget_s=10.0)
        cpu = {"value": ips, "unit": "images/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"{n} full steps of the same batch through oracle.fc_train_step ({sec * 1e3:.0f} ms "
                         "each; numpy's BLAS threads for the three fp64 products, single-threaded C for the "
                         "elementwise stages)"}
    flops = 6.0 * B * K * O
    nbytes = step_bytes(B, K, O)
    achieved = nbytes / (ms_max * 1e-3) / 1e9
    line = {"metric": "Algorithm 1 training step of a fully connected MINW layer: images/s",
            "value": replica_throughput(B, world, ms_max * 1e-3), "unit": "images/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": fc_train_config(world),
            "roofline": {"bound": "hbm", "kernel": "the whole step (7 launches: 3 operand passes, 3 bf16 "
                                                   "tensor-core products, the forward's K-slice sum, the "
                                                   "update inside the weight-gradient epilogue)",
                         "achieved": achieved, "peak": HBM_GBS, "unit": "GB/s",
                         "frac": achieved / HBM_GBS, "traffic": None, "bytes_per_step": nbytes,
                         "peak_basis": "measured HBM copy GB/s, of measured"},
            "tensor_tflops": flops / (ms_max * 1e-3) / 1e12,
            "cpu_baseline": cpu,
            "e2e": {"value": replica_throughput(B, world, e2e_sec), "unit": "images/s",
                    "h2d_bytes_per_step": int(4 * (A.numel() + G.numel())), "d2h_bytes_per_step": int(4 * g_in.numel())},
            "gpu_launches": 7 * args.steps, "clocks": clk.summary()}
    return line


# --------------------------------------------------------- conv training --

CONV_TRAIN_SHAPE = (256, 256, 16, 16, 256, 3, 1, 1)    # B, C, H, W, O, k, stride, pad: Model A's conv4
CONV_TRAIN_ALPHA, CONV_TRAIN_LR = 0.75, 1e-3


def conv_train_dims():
    B, C, H, W, O, k, s, p = CONV_TRAIN_SHAPE
    Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
    Hd, Wd = (Ho - 1) * s + 1 + (H + 2 * p - k) % s, (Wo - 1) * s + 1 + (W + 2 * p - k) % s
    return B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd


def conv_step_bytes():
    """Bytes the convolutional training step's launches move at least, launch
    by launch: the weight pass (W read; W^ written in the forward and the
    flipped layouts), the input's bf16 NHWC copy and its transposed patches
    (A read twice, both written), the forward product (bf16 input and W^
    read, a~ written), the gradient pass (a~ and g read; a_out, g~ as rows
    and as the spread NHWC image written), the input-gradient product (the
    spread image and the flipped W^ read, g_in written), the weight-gradient
    product (g~ rows and the patches read, the gradient written), and the
    update (W and the gradient read, W written)."""
    B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd = conv_train_dims()
    Op = (O + 63) // 64 * 64
    Kw, npix, x = C * k * k, B * Ho * Wo, B * C * H * W
    return float((4 * O * Kw + 2 * O * Kw + 2 * Kw * Op)
                 + (4 * x + 2 * x) + (4 * x + 2 * Kw * npix)
                 + (2 * x + 2 * O * Kw + 4 * O * npix)
                 + (8 * O * npix + 4 * O * npix + 2 * O * npix + 2 * B * Hd * Wd * Op)
                 + (2 * B * Hd * Wd * Op + 2 * C * k * k * Op + 4 * x)
                 + (2 * O * npix + 2 * Kw * npix + 4 * O * Kw)
                 + 12 * O * Kw)


def conv_min_bytes():
    """The step's irreducible traffic: A, W and g read once, a~ (a_pre),
    a_out, g_in and the updated W written once."""
    B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd = conv_train_dims()
    return float(4 * (B * C * H * W) * 2 + 4 * O * C * k * k * 2 + 4 * (B * O * Ho * Wo) * 3)


def conv_train_problem(rank=0):
    B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd = conv_train_dims()
    r = np.random.default_rng(37 + 1000 * rank)
    A = np.clip(r.standard_normal((B, C, H, W)), -1.5, 1.5).astype(np.float32)
    Wl = r.uniform(-1, 1, (O, C, k, k)).astype(np.float32)
    G = (r.standard_normal((B, O, Ho, Wo)) * 0.1).astype(np.float32)
    return A, Wl, G


def conv_train_config(world):
    B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd = conv_train_dims()
    return {"workload": f"conv_train_{C}to{O}_{H}x{W}_b{B}_a1w1", "batch_per_gpu": B, "global_batch": B * world,
            "layer": f"conv {k}x{k}/{s}/{p} {C} -> {O} at {H}x{W} (Model A's conv4), alpha {CONV_TRAIN_ALPHA}, "
                     f"lr {CONV_TRAIN_LR}, SGD + clip",
            "parallelism": f"replicas x{world} (no gradient all-reduce)", "l2": L2_NOTE}


def conv_train_oracle_rate(A, Wl, G, budget_s=10.0, images=2):
    """The oracle's convolutional training step (oracle.conv_train_step) on
    the first `images` images of the batch, repeated until budget_s seconds;
    returns (images/s, seconds per sub-batch step, steps)."""
    from oracle import oracle as Or
    from paper_2003_04296_gb300.inputs import DEFAULT_THR
    B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd = conv_train_dims()
    a, g = A[:images], G[:images]
    times = []
    t_start = time.perf_counter()
    while not times or time.perf_counter() - t_start < budget_s:
        t0 = time.perf_counter()
        Or.conv_train_step(a, Wl, g, CONV_TRAIN_ALPHA, CONV_TRAIN_LR, 1, DEFAULT_THR[1], s, p, (1, DEFAULT_THR[1]))
        times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    return images / sec, sec, len(times)


def run_reference_conv_train(args):
    A, Wl, G = conv_train_problem(0)
    steps = []
    for _ in range(args.steps):
        ips, sec, n = conv_train_oracle_rate(A, Wl, G, budget_s=0.0)
        steps.append(sec)
    sec = sum(steps) / len(steps)
    ips = 2 / sec
    line = {"metric": "Algorithm 1 training step of a convolutional MINW layer: images/s", "value": ips,
            "unit": "images/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": sec * 1e3, "higher_is_better": True, "impl": "reference", "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": conv_train_config(args.gpus),
            "cpu_baseline": {"value": ips, "unit": "images/s", "cores": 1, "kind": "oracle",
                             "sample": "each step: oracle.conv_train_step on 2 images of the batch (single-threaded "
                                       "C fp64 convolutions), scaled per image"},
            "e2e": {"value": ips, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_conv_train(args, rank, world, local_rank):
    """Algorithm 1's training step of Model A's conv4 (256 -> 256 channels,
    16 x 16, 3 x 3, batch 256, 1-bit weights and activations, alpha 0.75)
    through minw_conv_train_step: three bf16 tensor-core products (forward,
    input gradient, weight gradient) and five operand and update passes.
    Its roofline is HBM: the bytes its launches move at least
    (conv_step_bytes), over the step's event time; the fraction of the
    step's irreducible bytes (conv_min_bytes) is reported beside it."""
    import torch
    import __graft_entry__ as g
    if rank == 0:
        g.build()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    from paper_2003_04296_gb300 import minw
    from paper_2003_04296_gb300.inputs import DEFAULT_THR
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    B, C, H, W, O, k, s, p, Ho, Wo, Hd, Wd = conv_train_dims()
    A_np, W_np, G_np = conv_train_problem(rank)
    A, Wl, G = (torch.from_numpy(x).to(dev) for x in (A_np, W_np, G_np))
    a_out = torch.empty((B, O, Ho, Wo), device=dev)
    g_in = torch.empty((B, C, H, W), device=dev)
    ws = torch.empty(minw.minw_conv_train_workspace_bytes(B, C, H, W, O, k, k, s, p), dtype=torch.uint8, device=dev)
    qw, qa = minw.quant(1, DEFAULT_THR[1]), minw.quant(1, DEFAULT_THR[1])
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        minw.minw_conv_train_step(A, Wl, G, s, p, CONV_TRAIN_ALPHA, CONV_TRAIN_LR, qw, qa, a_out, g_in, ws)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    with ClockSampler(local_rank) as clk:
        for kk in range(args.steps):
            flush.zero_()
            e0[kk].record(stream)
            step()
            e1[kk].record(stream)
        torch.cuda.synchronize()
    ms_max = max_over_ranks(sum(e0[kk].elapsed_time(e1[kk]) for kk in range(args.steps)) / args.steps, world, dev)
    A_host = A.cpu().pin_memory()
    G_host = G.cpu().pin_memory()
    gin_host = torch.empty((B, C, H, W), dtype=torch.float32).pin_memory()
    e2e_s = []
    for kk in range(min(args.steps, 20) + 1):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        A.copy_(A_host, non_blocking=True)
        G.copy_(G_host, non_blocking=True)
        step()
        gin_host.copy_(g_in, non_blocking=True)
        torch.cuda.synchronize()
        if kk:
            e2e_s.append(time.perf_counter() - t0)
    e2e_sec = max_over_ranks(sum(e2e_s) / len(e2e_s), world, dev)
    if rank != 0:
        return None
    cpu = None
    if world == 1 and not args.skip_cpu:
        ips, sec, n = conv_train_oracle_rate(A_np, W_np, G_np, budget_s=10.0)
        cpu = {"value": ips, "unit": "images/s", "cores": 1, "kind": "oracle",
               "sample": f"{n} steps of oracle.conv_train_step on 2 images of the batch ({sec:.2f} s each; "
                         "single-threaded C fp64 convolutions), scaled per image"}
    flops = 6.0 * B * Ho * Wo * O * C * k * k
    nbytes = conv_step_bytes()
    achieved = nbytes / (ms_max * 1e-3) / 1e9
    line = {"metric": "Algorithm 1 training step of a convolutional MINW layer: images/s",
            "value": replica_throughput(B, world, ms_max * 1e-3), "unit": "images/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": conv_train_config(world),
            "roofline": {"bound": "hbm", "kernel": "the whole step (10 launches: weight, input and gradient "
                                                   "passes, 3 bf16 tensor-core products, the weight gradient's "
                                                   "slice sum, the update)",
                         "achieved": achieved, "peak": HBM_GBS, "unit": "GB/s",
                         "frac": achieved / HBM_GBS, "traffic": None, "bytes_per_step": nbytes,
                         "frac_of_irreducible_bytes": conv_min_bytes() / (ms_max * 1e-3) / 1e9 / HBM_GBS,
                         "irreducible_bytes": conv_min_bytes(),
                         "peak_basis": "measured HBM copy GB/s, of measured"},
            "tensor_tflops": flops / (ms_max * 1e-3) / 1e12,
            "cpu_baseline": cpu,
            "e2e": {"value": replica_throughput(B, world, e2e_sec), "unit": "images/s",
                    "h2d_bytes_per_step": int(4 * (A.numel() + G.numel())), "d2h_bytes_per_step": int(4 * g_in.numel())},
            "gpu_launches": 10 * args.steps, "clocks": clk.summary()}
    return line


def run_sweep(args, rank, world, local_rank):
    """One step: quantize the input to level codes and convolve it with the
    weight codes for each of the nine bit-width pairs (int32 accumulators),
    then the AQE forward and backward on the same tensor."""
    import torch
    import torch.distributed as dist
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    import __graft_entry__ as g
    if rank == 0:
        g.build()
    if world > 1:
        dist.barrier()
    from paper_2003_04296_gb300 import minw
    from paper_2003_04296_gb300.inputs import DEFAULT_THR, aqe_problem
    p = sweep_problem()
    B, C, H, W, O = 256, 512, 14, 14, 512
    x = torch.from_numpy(p["x"]).to(dev)
    w = torch.from_numpy(p["w"]).to(dev)
    ws = torch.from_numpy(p["w_scale"]).to(dev)
    g_np = aqe_problem(55, x.numel())["g"]
    gy = torch.from_numpy(g_np).to(dev)
    # level codes in both operand formats: E4M3 (one channel per byte, kind::f8f6f4) and E2M1 (two
    # channels per byte, kind::mxf4); each bit-width pair runs in the format and tiling measured fastest
    # for it below (E4M3, E2M1, or E2M1 as CTA pairs of 128-channel tiles)
    a8 = {(b, f): torch.empty((B, H, W, C if f == "e4m3" else C // 2), dtype=torch.uint8, device=dev)
          for b in (1, 2, 3) for f in ("e4m3", "e2m1")}
    w8 = {(b, f): torch.empty((O, 3, 3, C if f == "e4m3" else C // 2), dtype=torch.uint8, device=dev)
          for b in (1, 2, 3) for f in ("e4m3", "e2m1")}
    for b in (1, 2, 3):
        minw.minw_pack_weight_codes(w, minw.quant(b, DEFAULT_THR[b]), w8[(b, "e4m3")], channel_scale=ws)
        minw.minw_pack_weight_codes_e2m1(w, minw.quant(b, DEFAULT_THR[b]), w8[(b, "e2m1")], channel_scale=ws)
        minw.aqe_quantize_codes(x, minw.quant(b, DEFAULT_THR[b]), a8[(b, "e4m3")])
        minw.aqe_quantize_codes_e2m1(x, minw.quant(b, DEFAULT_THR[b]), a8[(b, "e2m1")])
    acc = torch.empty((B, O, H, W), dtype=torch.int32, device=dev)
    y = torch.empty_like(x)
    stream = torch.cuda.current_stream()
    FORMATS = [("e4m3", False), ("e2m1", False), ("e2m1", True)]

    def conv(ba, bw, fmt):
        f, pairs = fmt
        minw.minw_conv_block_codes_ex(a8[(ba, f)], B, C, H, W, ba, w8[(bw, f)], O, 3, 3, bw, 1, 1, 0, None, None,
                                      in_format=minw.CODES_E2M1 if f == "e2m1" else minw.CODES_E4M3,
                                      acc_out=acc, e2m1_pairs=pairs)

    # the measured choice: the least of three timed launches of each candidate, after one warm-up
    choice, cand_ms = {}, {}
    for ba, bw in SWEEP_PAIRS:
        times = []
        for fmt in FORMATS:
            conv(ba, bw, fmt)
            best = 1e30
            for _ in range(3):
                t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                t0.record(stream)
                conv(ba, bw, fmt)
                t1.record(stream)
                t1.synchronize()
                best = min(best, t0.elapsed_time(t1))
            times.append(best)
        cand_ms[f"a{ba}w{bw}"] = [round(t, 5) for t in times]
        choice[(ba, bw)] = FORMATS[int(np.argmin(times))]
    q_fmts = {b: sorted({choice[(ba, bw)][0] for ba, bw in SWEEP_PAIRS if ba == b}) for b in (1, 2, 3)}
    q_first = (1, q_fmts[1][0])
    # weight-only layer at the same shape (bf16 activations x 1-bit weights), timed beside the steps
    xb = torch.empty((B, H, W, C), dtype=torch.int16, device=dev)
    wb = torch.empty((O, 3, 3, C), dtype=torch.int16, device=dev)
    minw.minw_to_bf16_nhwc(x, xb)
    minw.minw_pack_weight_bf16(w, minw.quant(1, DEFAULT_THR[1]), wb, channel_scale=ws)
    yw = torch.empty((B, O, H, W), dtype=torch.float32, device=dev)
    sc1, sh0 = torch.ones(O, device=dev), torch.zeros(O, device=dev)
    gx = torch.empty_like(x)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def quantize(b, f):
        if f == "e2m1":
            minw.aqe_quantize_codes_e2m1(x, minw.quant(b, DEFAULT_THR[b]), a8[(b, f)])
        else:
            minw.aqe_quantize_codes(x, minw.quant(b, DEFAULT_THR[b]), a8[(b, f)])

    def step(ev=None):
        for b in (1, 2, 3):
            for f in q_fmts[b]:
                if ev is not None and (b, f) == q_first:
                    ev[12][0].record(stream)
                quantize(b, f)
                if ev is not None and (b, f) == q_first:
                    ev[12][1].record(stream)
        for i, (ba, bw) in enumerate(SWEEP_PAIRS):
            if ev is not None:
                ev[i][0].record(stream)
            conv(ba, bw, choice[(ba, bw)])
            if ev is not None:
                ev[i][1].record(stream)
        if ev is not None:
            ev[9][0].record(stream)
        minw.aqe_forward(x, y, 0.75, minw.quant(2, DEFAULT_THR[2]))
        if ev is not None:
            ev[9][1].record(stream)
        minw.aqe_backward(x, gy, gx, 0.75)
        if ev is not None:
            # outside the timed steps: the stochastic forward (Eq. our, z from Philox4x64-10)
            ev[10][0].record(stream)
            minw.aqe_forward_stochastic(x, y, 0.75, 2026, 0)
            ev[10][1].record(stream)
            ev[11][0].record(stream)
            minw.minw_conv2d_bf16(xb, B, C, H, W, wb, O, 3, 3, 1, 1, 1, 0, sc1, sh0, yw)
            ev[11][1].record(stream)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    e0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clk:
        for k in range(args.steps):
            flush.zero_()
            e0[k].record(stream)
            step()
            e1[k].record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
    ms = sum(e0[k].elapsed_time(e1[k]) for k in range(args.steps)) / args.steps
    ms_max = max_over_ranks(ms, world, dev)
    # per-kernel durations: the same steps again with events around the convolutions and the AQE forward
    conv_ms = np.zeros(len(SWEEP_PAIRS))
    aqe_ms = sto_ms = wo_ms = q_ms = 0.0
    for k in range(args.steps):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(13)]
        flush.zero_()
        step(ev)
        torch.cuda.synchronize()
        conv_ms += np.array([ev[i][0].elapsed_time(ev[i][1]) for i in range(9)])
        aqe_ms += ev[9][0].elapsed_time(ev[9][1])
        sto_ms += ev[10][0].elapsed_time(ev[10][1])
        wo_ms += ev[11][0].elapsed_time(ev[11][1])
        q_ms += ev[12][0].elapsed_time(ev[12][1])
    conv_ms /= args.steps
    q_ms /= args.steps
    aqe_ms /= args.steps
    sto_ms /= args.steps
    wo_ms /= args.steps

    # end to end: the fp32 input from pinned host memory, the step, the last accumulators back to the host
    x_host = torch.from_numpy(p["x"]).pin_memory()
    acc_host = torch.empty(acc.shape, dtype=torch.int32).pin_memory()
    e2e_steps = min(args.steps, 20)
    e2e_s = []
    for k in range(e2e_steps + 1):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        x.copy_(x_host, non_blocking=True)
        step()
        acc_host.copy_(acc, non_blocking=True)
        torch.cuda.synchronize()
        if k:
            e2e_s.append(time.perf_counter() - t0)
    e2e_sec = max_over_ranks(sum(e2e_s) / len(e2e_s), world, dev)
    if rank != 0:
        return None

    mac = B * H * W * O * C * 9
    value = replica_throughput(2.0 * mac * len(SWEEP_PAIRS), world, ms_max * 1e-3) / 1e12
    achieved = 2.0 * mac * len(SWEEP_PAIRS) / (conv_ms.sum() * 1e-3) / 1e12
    kinds = [choice[pr][0] for pr in SWEEP_PAIRS]
    roofline = tensor_roofline([2.0 * mac] * len(SWEEP_PAIRS), kinds, [float(v) for v in conv_ms])
    roofline["kernel"] += " (9 bit-width pairs, int32 accumulators out)"
    roofline["pair_formats"] = {f"a{ba}w{bw}": choice[(ba, bw)][0] + (" CTA pairs" if choice[(ba, bw)][1] else "")
                                for ba, bw in SWEEP_PAIRS}
    roofline["candidate_ms"] = {"order": ["e4m3", "e2m1", "e2m1 CTA pairs of 128-channel tiles"], **cand_ms}
    # the A2 step: fp32 NCHW in, level codes out (4 + 1/2 bytes per element for E2M1, 4 + 1 for E4M3)
    q_bytes = (4.5 if q_first[1] == "e2m1" else 5.0) * x.numel()
    quant_roof = {"bound": "hbm", "kernel": f"quantize_codes_kernel<{q_first[1].upper()}> (1-bit)", "ms": round(q_ms, 5),
                  "achieved": q_bytes / (q_ms * 1e-3) / 1e9, "peak": HBM_GBS, "unit": "GB/s",
                  "frac": q_bytes / (q_ms * 1e-3) / 1e9 / HBM_GBS, "algorithmic_bytes": q_bytes,
                  "peak_basis": "measured copy bandwidth, of measured"}
    aqe_bytes = 8.0 * x.numel()
    aqe_roof = {"bound": "hbm", "kernel": "aqe_forward_kernel", "achieved": aqe_bytes / (aqe_ms * 1e-3) / 1e9,
                "peak": HBM_GBS, "unit": "GB/s", "frac": aqe_bytes / (aqe_ms * 1e-3) / 1e9 / HBM_GBS,
                "algorithmic_bytes": aqe_bytes, "peak_basis": "measured copy bandwidth, of measured"}
    sto_roof = {"bound": "hbm", "kernel": "aqe_forward_stochastic_kernel (Eq. our, Philox4x64-10 noise)",
                "achieved": aqe_bytes / (sto_ms * 1e-3) / 1e9, "peak": HBM_GBS, "unit": "GB/s",
                "frac": aqe_bytes / (sto_ms * 1e-3) / 1e9 / HBM_GBS, "algorithmic_bytes": aqe_bytes,
                "peak_basis": "measured copy bandwidth, of measured"}
    wo_tf = 2.0 * mac / (wo_ms * 1e-3) / 1e12
    wonly = {"kernel": "conv_tc_kernel<0, true, true> (tcgen05 kind::f16, CTA pairs: bf16 activations x 1-bit weights)",
             "ms": round(wo_ms, 5), "achieved": wo_tf, "peak": BF16_TFLOPS, "unit": "TFLOP/s",
             "frac": wo_tf / BF16_TFLOPS, "peak_basis": "measured dense bf16 TFLOP/s (burst), of measured"}
    cpu = None
    if world == 1 and not args.skip_cpu:
        from oracle import oracle as Or
        xs = p["x"][:1]
        a_lv = Or.quantize(xs, 1, DEFAULT_THR[1])
        w_lv = Or.quantize(p["w"], 1, DEFAULT_THR[1], p["w_scale"])
        t0 = time.perf_counter()
        n = 0
        while True:
            Or.conv2d_levels(a_lv, w_lv, 1, 1, 1, 1)
            n += 1
            if time.perf_counter() - t0 > args.cpu_seconds / 2:
                break
        dt = time.perf_counter() - t0
        cpu = {"value": 2.0 * (mac / B) * n / dt / 1e12, "unit": "effective TOPS", "cores": 1, "kind": "oracle",
               "sample": f"{n} single-image 1-bit x 1-bit convolutions (fp64 oracle, {dt:.1f} s)"}
    line = {"metric": METRIC, "value": value, "unit": "effective TOPS (2 x MAC / s)", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "+".join(sorted(set(kinds))), "data": "synthetic",
            "config": sweep_config(world),
            "conv_ms": [round(v, 5) for v in conv_ms.tolist()], "aqe_forward_ms": round(aqe_ms, 5),
            "aqe_stochastic_ms": round(sto_ms, 5),
            "roofline": roofline, "aqe_roofline": aqe_roof, "aqe_stochastic_roofline": sto_roof,
            "quantize_roofline": quant_roof,
            "weight_only_bf16": wonly, "cpu_baseline": cpu,
            "e2e": {"value": 2.0 * mac * len(SWEEP_PAIRS) * world / e2e_sec / 1e12, "unit": "effective TOPS",
                    "h2d_bytes_per_step": int(x_host.numel() * 4), "d2h_bytes_per_step": int(acc_host.numel() * 4)},
            "gpu_launches": (sum(len(v) for v in q_fmts.values()) + len(SWEEP_PAIRS) + 2) * args.steps,
            "clocks": clk.summary()}
    return line


def run_peaks(args, rank, world, local_rank):
    """The pipe rates behind the per-shape choice of path
    (minw_measure_pipe_rates), with per-SM-per-clock figures and the resulting
    peak of each path for a 1-bit x 1-bit convolution."""
    import torch
    torch.cuda.set_device(local_rank)
    import __graft_entry__ as g
    g.build()
    from paper_2003_04296_gb300 import minw
    r = minw.minw_measure_pipe_rates()
    if rank != 0:
        return None
    mhz = r["sm_clock_mhz"]
    per_clk = lambda v: v / (SMS * mhz * 1e6)
    paths = {"popcount (XOR + POPC, 32 binary MACs per popc)": 2.0 * 32 * r["popc_per_s"],
             "mma.sync b1 xor.popc": 2.0 * r["bmma_b1_mac_per_s"],
             "mma.sync s8": 2.0 * r["imma_s8_mac_per_s"],
             "tcgen05 kind::f8f6f4 E4M3 (N=256)": r["tc_e4m3_flop_per_s"][1],
             "tcgen05 kind::mxf4 E2M1 (N=256)": r["tc_e2m1_flop_per_s"][1]}
    return {"metric": "pipe rates of the quantized convolution's candidate paths", "n_gpus": 1,
            "value": r["tc_e2m1_flop_per_s"][1] / 1e12, "unit": "TFLOP/s (tcgen05 E2M1, N = 256)",
            "higher_is_better": True, "data": "synthetic", "config": {"workload": "pipe_rates"},
            "rates": r,
            "per_sm_per_clock": {"popc": per_clk(r["popc_per_s"]), "bmma_b1_mac": per_clk(r["bmma_b1_mac_per_s"]),
                                 "imma_s8_mac": per_clk(r["imma_s8_mac_per_s"]),
                                 "tc_e4m3_flop_n256": per_clk(r["tc_e4m3_flop_per_s"][1]),
                                 "tc_e2m1_flop_n256": per_clk(r["tc_e2m1_flop_per_s"][1]),
                                 "tc_bf16_flop_n256": per_clk(r["tc_bf16_flop_per_s"][1])},
            "binary_conv_tops_by_path": {k: v / 1e12 for k, v in paths.items()}}


def other_configs(args, rank, world, local_rank):
    """The default run's summary of the other benchmark workloads (each with
    fewer steps than its own run, no CPU baseline): the single convolution,
    the ConvNet at 2-bit activations with 1- and 2-bit weights, ResNet-18, the
    weight-only ResNet-110 and DenseNet-100 of Table III, and the bit-width
    sweep."""
    import copy
    out = {}
    jobs = [("conv1", run_conv1, dict(workload="conv1", steps=3000)),
            ("cifar_convnet_a2w1", run_gpu, dict(workload="cifar_convnet", bits_a=2, bits_w=1, steps=1500)),
            ("cifar_convnet_a2w2", run_gpu, dict(workload="cifar_convnet", bits_a=2, bits_w=2, steps=1500)),
            ("resnet18_a3w3", run_gpu, dict(workload="resnet18", steps=200)),
            ("wresnet110_w3", run_gpu, dict(workload="wresnet110", steps=200)),
            ("densenet100_w3", run_gpu, dict(workload="wdense100", steps=100)),
            ("sweep", run_sweep, dict(workload="sweep", steps=40))]
    for name, fn, ch in jobs:
        a = copy.copy(args)
        for k, v in ch.items():
            setattr(a, k, v)
        a.skip_cpu = True
        r = fn(a, rank, world, local_rank)
        if r is None:
            continue
        roof = r.get("roofline", {})
        out[name] = {"workload": r["config"]["workload"], "value": r["value"], "unit": r["unit"],
                     "ms_per_step": r["ms_per_step"], "steps": r["steps"], "dtype": r["dtype"],
                     "roofline_frac": roof.get("frac"), "roofline_frac_probe": roof.get("frac_probe"),
                     "roofline_kernel": roof.get("kernel"), "e2e": r.get("e2e", {}).get("value"),
                     "clocks": r.get("clocks")}
        for extra in ("layer_ms", "conv_ms"):
            if extra in r:
                out[name][extra] = r[extra]
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (defaults give about half a second of timed work, so that the clock "
                         "sampler sees several samples under load)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["minw", "reference"], default="minw")
    ap.add_argument("--workload", choices=["cifar_convnet", "resnet18", "wresnet110", "wdense100", "sweep",
                                           "fc_train", "conv_train", "conv1", "peaks"],
                    default="cifar_convnet")
    ap.add_argument("--bits-a", type=int, default=1, help="CIFAR ConvNet activation bits")
    ap.add_argument("--bits-w", type=int, default=1, help="CIFAR ConvNet weight bits")
    ap.add_argument("--model", choices=["A", "B", "C", "D"], default="A",
                    help="CIFAR ConvNet of Sec. IV-B (B-D: fewer channels)")
    ap.add_argument("--bits-a-resnet", type=int, default=3)
    ap.add_argument("--bits-w-resnet", type=int, default=3)
    ap.add_argument("--variant", type=int, default=0, help="0 auto, 1 popcount, 2 tensor cores")
    ap.add_argument("--layer-variants", default=None,
                    help="comma-separated kernel request per layer (the layer_variants of an earlier run): "
                         "replays that measured plan instead of measuring at creation")
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    ap.add_argument("--skip-cpu", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="default run: skip the summary of the other benchmark workloads")
    args = ap.parse_args()
    default_run = args.steps is None and args.workload == "cifar_convnet"
    if args.steps is None:
        args.steps = {"cifar_convnet": 4000, "resnet18": 400, "wresnet110": 500, "wdense100": 300, "sweep": 100,
                      "fc_train": 2000,
                      "conv_train": 500,
                      "conv1": 1000, "peaks": 1}[args.workload]

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank)
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    try:
        runner = {"sweep": run_sweep, "fc_train": run_fc_train, "conv_train": run_conv_train, "conv1": run_conv1,
                  "peaks": run_peaks}.get(args.workload, run_gpu)
        line = runner(args, rank, world, local_rank)
        if line is not None and default_run and world == 1 and not args.no_configs:
            line["configs"] = other_configs(args, rank, world, local_rank)
        if line is not None:
            print(json.dumps(line), flush=True)
        return 0
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
