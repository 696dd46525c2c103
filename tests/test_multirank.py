"""The multi-GPU path of bench.py, on CPU with two gloo ranks.

Under torchrun every rank verifies its own batch of sequences (weak scaling; the
sequences are independent, so there is no collective on the data path), the
step time is the slowest rank's (all_reduce MAX), and the reported throughput is
all ranks' positions over that time.  This checks those host-side pieces; the
kernels themselves need a GPU.
"""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


class _Args:
    config = 0
    rule = None
    alpha = None
    B = None
    gamma = None
    beta = 1.0
    temperature = None


def _worker(rank, world, port, queue):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = bench.max_over_ranks(1.0 + rank, world, "cpu")
    w, _ = bench.workload_from(_Args, rank)
    queue.put((rank, ms, float(abs(w.draft).sum()), bench.whole_job_rate(w.B * w.gamma, world, ms)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, queue)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    res = sorted(queue.get(timeout=10) for _ in range(2))
    assert res[0][1] == res[1][1] == 2.0          # both ranks report the slowest rank's time
    assert res[0][2] != res[1][2]                 # each rank verifies its own sequences
    # cfg0 holds 1 sequence of 4 drafts per rank: 8 positions in 2 ms
    assert res[0][3] == pytest.approx(2 * 1 * 4 / 2e-3)
