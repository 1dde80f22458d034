"""The multi-GPU path of the bench as independent batch replicas (no data-path
collective), on CPU with two gloo ranks: each rank draws its own images, the
job's time is the slowest rank's (every rank learns it), the whole-job
throughput counts all ranks' images, and the oracle forward of each rank's
images is unaffected by the other rank."""
import os
import socket
import sys
import types

import numpy as np
import pytest

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    try:
        dist.init_process_group("gloo", rank=rank, world_size=world)
        import bench
        from oracle import network as N
        from paper_2003_04296_gb300 import inputs as I
        args = types.SimpleNamespace(bits_a=1, bits_w=1, bits_a_resnet=3, bits_w_resnet=3)
        wl = bench.Workload("cifar_convnet", args)
        x = wl.images(rank)
        slow = bench.max_over_ranks(0.25 + 0.5 * rank, world, "cpu")       # per-rank step seconds
        ips = bench.replica_throughput(wl.batch, world, slow)
        # a small net on two images of this rank's batch: the replica's own forward
        p = I.convnet_params(5, widths=(32, 32, 32, 32), pools=(False, True, False, True), fcs=(32,), hw=8)
        xs = I.convnet_input(6 + 1000 * rank, 2, hw=8)
        logits = N.convnet_forward(p, xs)
        gathered = [torch.zeros(4, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(gathered, torch.tensor(x.reshape(-1)[:4].astype(np.float64)))
        dist.barrier()
        dist.destroy_process_group()
        q.put((rank, slow, ips, float(x.sum()), [g.numpy().tolist() for g in gathered], logits.tolist(),
               xs.tolist()))
    except Exception as e:  # reported to the parent
        q.put((rank, repr(e)))


def test_two_replicas_gloo():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(2):
        item = q.get(timeout=300)
        res[item[0]] = item
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        assert len(res[r]) == 7, res[r]
    # the slowest rank's time reaches both ranks; throughput counts both batches
    assert res[0][1] == res[1][1] == 0.75
    assert res[0][2] == res[1][2] == pytest.approx(2 * 256 / 0.75)
    # independent replicas: different images per rank, each rank sees both in the gather
    assert res[0][3] != res[1][3]
    assert res[0][4] == res[1][4] and res[0][4][0] != res[0][4][1]
    # each replica's forward equals the oracle run alone on its own images
    from oracle import network as N
    from paper_2003_04296_gb300 import inputs as I
    p = I.convnet_params(5, widths=(32, 32, 32, 32), pools=(False, True, False, True), fcs=(32,), hw=8)
    for r in range(2):
        xs = np.array(res[r][6], dtype=np.float32)
        assert np.array_equal(np.array(res[r][5]), N.convnet_forward(p, xs))
