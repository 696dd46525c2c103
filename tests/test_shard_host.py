"""Host logic of the vocabulary-sharded step (paper_2405_19261_gb300/sharded.py)
on CPU: the shard partition, the phase order, and the all-gather of the
phase messages in rank order -- in one process (LocalExchange) and across two
gloo processes (DistExchange, the path NCCL takes between GPUs).  The kernels
need a GPU; here each phase is a stand-in whose message names its rank and
phase, and which checks the gathered messages it receives."""
import os
import socket
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2405_19261_gb300 import sharded  # noqa: E402

SIZES = {1: 48, 2: 16, 3: 16, 4: 8, 5: 8}


class PhaseProbe:
    """Stands in for ShardRank: message k of rank r is SIZES[k] bytes of
    10 k + r; each phase asserts that it received every rank's previous
    message in rank order, and records the phases it ran."""

    def __init__(self, rank, W):
        self.rank, self.W, self.log = rank, W, []

    def _msg(self, k):
        return torch.full((SIZES[k],), 10 * k + self.rank, dtype=torch.uint8)

    def _expect(self, g, k):
        want = torch.cat([torch.full((SIZES[k],), 10 * k + r, dtype=torch.uint8) for r in range(self.W)])
        assert torch.equal(g, want), (k, g)

    def pass1(self, d, t, tokens, T, rule, stream=None):
        self.log.append("pass1")
        return self._msg(1)

    def decide(self, d, t, g1, tokens, uniforms, rule, alpha, T, stream=None):
        self._expect(g1, 1)
        self.log.append("decide")
        return self._msg(2)

    def tv(self, d, t, g2, rule, alpha, T, stream=None):
        assert rule == 2  # OPT only: the lower bound's parts were exchanged
        self._expect(g2, 2)
        self.log.append("tv")
        return self._msg(3)

    def accept(self, d, t, g3, uniforms, rule, alpha, T, stream=None):
        if rule == 2:  # OPT: the D_TV parts were exchanged
            self._expect(g3, 3)
        else:
            assert g3 is None
        self.log.append("accept")
        return self._msg(4)

    def draw(self, d, t, g4, uniforms, T, stream=None):
        self._expect(g4, 4)
        self.log.append("draw")
        return self._msg(5)

    def finish(self, g5, stream=None):
        self._expect(g5, 5)
        self.log.append("finish")
        return torch.tensor([self.W]), g5.clone()


def test_shard_bounds():
    for V, W in ((256000, 1), (256000, 2), (256000, 3), (256000, 8), (256000, 16), (32128, 16), (1001, 7)):
        for align in (1, 8):
            try:
                b = sharded.shard_bounds(V, W, align)
            except ValueError:
                assert align == 8 and V == 1001  # 7 shards of a multiple of 8 do not fit evenly
                continue
            assert b[0] == 0 and b[-1] == V and len(b) == W + 1
            assert all(b[r + 1] > b[r] for r in range(W))
            assert all(v % align == 0 for v in b[1:-1])
            widths = [b[r + 1] - b[r] for r in range(W)]
            assert max(widths) - min(widths) <= W * align
    with pytest.raises(ValueError):
        sharded.shard_bounds(10, 17)
    with pytest.raises(ValueError):
        sharded.shard_bounds(5, 8)


@pytest.mark.parametrize("rule", ["opt", "diff"])
def test_phases_in_one_process(rule):
    W = 3
    ranks = [PhaseProbe(r, W) for r in range(W)]
    out = sharded.sharded_step(ranks, [(None, None)] * W, None, None, rule, 0.2, 1.0, sharded.LocalExchange())
    phases = ["pass1", "decide"] + (["tv"] if rule == "opt" else []) + ["accept", "draw", "finish"]
    for r in ranks:
        assert r.log == phases
    assert all(torch.equal(o[1], out[0][1]) for o in out)


def test_rules_outside_table1_are_refused():
    with pytest.raises(ValueError):
        sharded.sharded_step([PhaseProbe(0, 1)], [(None, None)], None, None, "token_v3", 0.3, 1.0,
                             sharded.LocalExchange())


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, rule, queue):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    from paper_2405_19261_gb300 import sharded as sh
    dist.init_process_group("gloo", rank=rank, world_size=world)
    probe = PhaseProbe(rank, world)
    out = sh.sharded_step([probe], [(None, None)], None, None, rule, 0.2, 1.0, sh.DistExchange())
    queue.put((rank, probe.log, out[0][1].tolist()))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("rule", ["opt", "chow"])
def test_two_gloo_ranks_exchange_in_rank_order(rule):
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, rule, queue)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    res = sorted(queue.get(timeout=10) for _ in range(2))
    phases = ["pass1", "decide"] + (["tv"] if rule == "opt" else []) + ["accept", "draw", "finish"]
    for rank, log, final in res:
        assert log == phases
    assert res[0][2] == res[1][2]  # both ranks hold the same gathered result
