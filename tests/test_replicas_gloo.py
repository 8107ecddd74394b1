"""The N-GPU benchmark's replica bookkeeping (paper_2609_16742_gb300/replicas.py)
on two gloo ranks on CPU: every rank takes disjoint input images, timings
reduce to the maximum over ranks, the whole-job throughput counts every
rank's images."""
import os
import socket

import pytest

from paper_2609_16742_gb300 import replicas


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        t = replicas.reduce_max(10.0 + 2.5 * rank, dist, "cpu")
        q.put((rank, t, replicas.input_slices(rank, 256)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        got = sorted(q.get(timeout=120) for _ in procs)
    finally:
        for p in procs:
            p.join(timeout=60)
    assert [p.exitcode for p in procs] == [0, 0]
    assert [t for _, t, _ in got] == [12.5, 12.5]             # the slower rank's time on both
    images = [set(range(f, f + 256)) for _, _, sl in got for f in sl]
    assert len(images) == 4 and len(set().union(*images)) == 4 * 256   # disjoint batches


def test_one_process_and_throughput():
    assert replicas.reduce_max(3.25) == 3.25
    assert replicas.input_slices(0, 128) == [0, 128]
    assert replicas.input_slices(3, 128, per_rank=2) == [768, 896]
    assert replicas.job_throughput(4, 256, 20, 0.5) == pytest.approx(4 * 256 * 20 / 0.5)
