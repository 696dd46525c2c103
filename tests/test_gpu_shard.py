"""Vocabulary-sharded verification (include/sc_shard.h) against the fp64 oracle
(GPU only).

The W ranks run on one GPU as one process (sharded.emulated_step): each rank's
kernels read its shard as a view of the full logits, and the messages between
the phases are concatenated on the device where a multi-GPU run would
all-gather them.  The kernels and the arithmetic are those of a W-GPU run.
The sharded step must reach the oracle's decisions and tokens -- the oracle
knows nothing of shards -- on every sequence the oracle does not flag, for
every W, partition, rule and logit type; every rank must hold the same
outputs; and it must agree with the single-GPU kernel (sc_verify).
"""
import numpy as np
import pytest

import oracle
from paper_2405_19261_gb300.workloads import config, synthetic

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sh():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2405_19261_gb300 import sharded
    sharded.lib()
    return sharded


def run_sharded(sh, w, bounds, rule=None, alpha=None, check_ranks=True):
    import torch
    from paper_2405_19261_gb300 import binding
    d, t, x, u = binding.to_device(w)
    na, nt, ranks = sh.emulated_step(d, t, x, u, rule or w.rule, w.alpha if alpha is None else alpha,
                                     w.temperature, bounds)
    torch.cuda.synchronize()
    out = na.cpu().numpy().copy(), nt.cpu().numpy().copy()
    status = [int(r.status.item()) for r in ranks]
    if check_ranks:  # every rank holds the same outputs and the same status
        for r in ranks:
            assert np.array_equal(r.num_accepted.cpu().numpy(), out[0])
            assert np.array_equal(r.next_token.cpu().numpy(), out[1])
        assert len(set(status)) == 1, status
    return out[0], out[1], status[0]


def assert_sharded_parity(w, got, ref, min_compared=None):
    na, nt, status = got
    assert status == 0, f"{w.name}: device status {status}"
    ok = ~ref.flagged
    if min_compared is None:  # a handful of sequences may all sit near one decision
        min_compared = 0.8 if w.B >= 32 else 0.5
    assert ok.mean() >= min_compared, f"{w.name}: only {ok.sum()} of {w.B} sequences comparable"
    bad = np.nonzero(ok & ((na != ref.num_accepted) | (nt != ref.next_token)))[0]
    assert len(bad) == 0, (f"{w.name}: {len(bad)} unflagged mismatches, first b={bad[:5]}, "
                           f"gpu={na[bad[:5]]},{nt[bad[:5]]} oracle={ref.num_accepted[bad[:5]]},"
                           f"{ref.next_token[bad[:5]]}")
    return int(ok.sum())


_held = {}
_ref = {}


def held(key, make):
    if key not in _held:
        _held.clear()
        _held[key] = make()
    return _held[key]


@pytest.mark.parametrize("W", [1, 2, 3, 4, 8, 16])
@pytest.mark.parametrize("rule,alpha", [("chow", 0.5), ("diff", 0.1), ("opt", 0.2), ("opt", 0.0),
                                        ("always", 0.0), ("never", 0.0)])
def test_t5_shape_every_shard_count(sh, W, rule, alpha):
    # cfg1's shape (B=8, gamma=5, V=32128 bf16) under every rule of Table 1 and
    # SpecDecode's delta = 1; 16 shards of 2008 tokens down to one of 32128
    w = held(("cfg1",), lambda: config(1)).with_rule(rule, alpha)
    ref = oracle.verify_workload(w)
    got = run_sharded(sh, w, sh.shard_bounds(w.V, W))
    assert_sharded_parity(w, got, ref)


@pytest.mark.parametrize("W", [2, 4])
@pytest.mark.parametrize("rule", ["chow", "diff", "opt"])
def test_gemma_shape_every_sequence(sh, W, rule):
    # a 256k-vocabulary sweep point (B=64, gamma=8), every sequence
    alpha = {"chow": 0.5, "diff": 0.1, "opt": 0.2}[rule]
    w = held(("g64",), lambda: config(4, B=64, gamma=8)).with_rule(rule, alpha)
    ref = oracle.verify_workload(w)
    n = assert_sharded_parity(w, run_sharded(sh, w, sh.shard_bounds(w.V, W)), ref)
    print(f"{w.name} W={W}: {n} of {w.B} compared")


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("bounds", [[0, 5001, 20000, 32128], [0, 1, 32127, 32128], [0, 16000, 16003, 32128]])
def test_ragged_partitions(sh, dtype, bounds):
    # shard starts that are not 16-byte aligned (element-by-element loads),
    # one-token shards, and shards narrower than a slice or a segment
    w = synthetic(12, 4, 32128, dtype=dtype, kind="gauss", sigma=0.6, rule="opt", alpha=0.3, seed=5)
    ref = oracle.verify_workload(w)
    assert_sharded_parity(w, run_sharded(sh, w, bounds), ref)


@pytest.mark.parametrize("W", [1, 2, 3])
def test_ragged_vocabulary(sh, W):
    # V not a multiple of 8 (the rows themselves are unaligned), f32 and bf16
    for dtype in ("f32", "bf16"):
        w = synthetic(6, 3, 1001, dtype=dtype, kind="gauss", sigma=0.8, rule="diff", alpha=0.05, seed=7)
        ref = oracle.verify_workload(w)
        assert_sharded_parity(w, run_sharded(sh, w, sh.shard_bounds(w.V, W, align=1)), ref)


def test_temperature_and_planted_rejections(sh):
    # cfg3: T = 0.7, per-row target noise, about half the sequences with a
    # certain early rejection; 2 and 4 shards
    w = held(("cfg3",), lambda: config(3))
    ref = oracle.verify_workload(w)
    for W in (2, 4):
        na, nt, st = run_sharded(sh, w, sh.shard_bounds(w.V, W))
        assert_sharded_parity(w, (na, nt, st), ref)
        f = w.forced >= 0
        assert np.all(na[f] <= w.forced[f])


@pytest.mark.slow
@pytest.mark.parametrize("W", [2, 4, 8])
def test_largest_sweep_point_every_sequence(sh, W):
    # cfg4 B=512 gamma=8 OPT 0.2 (4.46 GB of logits), every sequence, and the
    # single-GPU kernel's outputs on the same logits
    import torch
    from paper_2405_19261_gb300 import binding
    w = held(("g512",), lambda: config(4, B=512, gamma=8))
    if _ref.get("g512") is None or _ref["g512"][0] is not w:
        _ref["g512"] = (w, oracle.verify_workload(w))
    ref = _ref["g512"][1]
    na, nt, st = run_sharded(sh, w, sh.shard_bounds(w.V, W))
    n = assert_sharded_parity(w, (na, nt, st), ref)
    d, t, x, u = binding.to_device(w)
    na1, nt1 = binding.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature)
    torch.cuda.synchronize()
    ok = ~ref.flagged
    assert np.array_equal(na1.cpu().numpy()[ok], na[ok]) and np.array_equal(nt1.cpu().numpy()[ok], nt[ok])
    print(f"{w.name} W={W}: {n} of {w.B} compared, flagged {int(ref.flagged.sum())}")


def test_matches_the_single_gpu_kernel(sh):
    # the same logits through sc_verify and through 3 shards: identical outputs
    # on every sequence the oracle does not flag
    import torch
    from paper_2405_19261_gb300 import binding
    w = synthetic(48, 6, 100000, dtype="bf16", kind="zipf", sigma=0.9, rule="opt", alpha=0.3, seed=11)
    ref = oracle.verify_workload(w)
    na, nt, _ = run_sharded(sh, w, sh.shard_bounds(w.V, 3))
    d, t, x, u = binding.to_device(w)
    na1, nt1 = binding.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature)
    torch.cuda.synchronize()
    ok = ~ref.flagged
    assert np.array_equal(na1.cpu().numpy()[ok], na[ok])
    assert np.array_equal(nt1.cpu().numpy()[ok], nt[ok])


def test_repeated_steps_reuse_the_buffers(sh):
    # two different batches through the same rank objects: the second step's
    # outputs depend only on its own inputs
    import torch
    from paper_2405_19261_gb300 import binding
    bounds = sh.shard_bounds(32128, 2)
    ranks = None
    for seed in (21, 22):
        w = synthetic(8, 5, 32128, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.2, seed=seed)
        d, t, x, u = binding.to_device(w)
        na, nt, ranks = sh.emulated_step(d, t, x, u, w.rule, w.alpha, w.temperature, bounds, ranks=ranks)
        torch.cuda.synchronize()
        ref = oracle.verify_workload(w)
        assert_sharded_parity(w, (na.cpu().numpy(), nt.cpu().numpy(), 0), ref)


def test_data_errors_set_status_and_defined_outputs(sh):
    # a draft token outside [0, V), a uniform outside [0, 1) and a NaN logit in
    # three sequences (each on the shard that holds it): those sequences get
    # num_accepted = 0, next_token = -1 and their status bits on every rank;
    # the other sequences are unaffected
    from paper_2405_19261_gb300 import binding
    w = synthetic(8, 4, 32128, dtype="f32", kind="gauss", sigma=0.5, rule="diff", alpha=0.1, seed=3)
    ref = oracle.verify_workload(w)
    w.tokens = w.tokens.copy()
    w.uniforms = w.uniforms.copy()
    w.target = w.target.copy()
    w.tokens[1, 2] = w.V + 5
    w.uniforms[3, 0] = 1.0
    w.target[5, 1, 30000] = np.nan
    na, nt, st = run_sharded(sh, w, sh.shard_bounds(w.V, 2))
    assert st == binding.DEV_BAD_TOKEN | binding.DEV_BAD_UNIFORM | binding.DEV_BAD_LOGIT
    for b in (1, 3, 5):
        assert na[b] == 0 and nt[b] == -1
    keep = np.array([b not in (1, 3, 5) for b in range(w.B)]) & ~ref.flagged
    assert np.array_equal(na[keep], ref.num_accepted[keep]) and np.array_equal(nt[keep], ref.next_token[keep])


def test_masked_logits(sh):
    # -inf logits (a masked vocabulary tail on the last shard, and a masked
    # draft-token target logit, p(x) = 0 < q(x)) are probability 0, as in the oracle
    w = synthetic(8, 4, 32128, dtype="f32", kind="gauss", sigma=0.5, rule="always", alpha=0.0, seed=9)
    w.draft = w.draft.copy()
    w.target = w.target.copy()
    w.draft[:, :, 31000:] = -np.inf
    w.target[:, :, 31000:] = -np.inf
    w.tokens = np.minimum(w.tokens, 30999).astype(np.int32)
    w.target[2, 0, w.tokens[2, 0]] = -np.inf
    ref = oracle.verify_workload(w)
    got = run_sharded(sh, w, sh.shard_bounds(w.V, 4))
    assert_sharded_parity(w, got, ref)
    assert got[0][2] == 0


def test_graph_replay_matches_the_eager_step(sh):
    # the step captured as one CUDA graph (what bench.py --vocab-shards times):
    # replays with new inputs copied into the captured tensors give the eager
    # step's outputs and the oracle's
    import torch
    from paper_2405_19261_gb300 import binding
    bounds = sh.shard_bounds(32128, 3)
    w0 = synthetic(16, 5, 32128, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.2, seed=41)
    d, t, x, u = binding.to_device(w0)
    G = sh.EmulatedGraph(d, t, x, u, "opt", 0.2, 1.0, bounds)
    for seed in (42, 43):
        w = synthetic(16, 5, 32128, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.2, seed=seed)
        d1, t1, x1, u1 = binding.to_device(w)
        d.copy_(d1), t.copy_(t1), x.copy_(x1), u.copy_(u1)
        na, nt = G.replay()
        torch.cuda.synchronize()
        got = (na.cpu().numpy().copy(), nt.cpu().numpy().copy())
        na2, nt2, _ = sh.emulated_step(d1, t1, x1, u1, "opt", 0.2, 1.0, bounds)
        torch.cuda.synchronize()
        assert np.array_equal(got[0], na2.cpu().numpy()) and np.array_equal(got[1], nt2.cpu().numpy())
        assert_sharded_parity(w, (got[0], got[1], 0), oracle.verify_workload(w))


def _nccl_rank(port, queue):
    # one rank of a one-GPU NCCL process group: the step through DistExchange
    # (NCCL all-gathers of the device messages) and through LocalExchange
    import os
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK="0", WORLD_SIZE="1",
                      NCCL_NVLS_ENABLE="0")
    import torch
    import torch.distributed as dist
    from paper_2405_19261_gb300 import binding, sharded
    try:
        torch.cuda.set_device(0)
        dist.init_process_group("nccl", rank=0, world_size=1)
        w = synthetic(16, 5, 32128, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.2, seed=51)
        d, t, x, u = binding.to_device(w)
        res = {}
        for name, ex in (("nccl", sharded.DistExchange()), ("local", sharded.LocalExchange())):
            r = sharded.ShardRank(w.B, w.gamma, [0, w.V], 0, d.dtype, d.device)
            [(na, nt)] = sharded.sharded_step([r], [(d, t)], x, u, "opt", 0.2, 1.0, ex)
            torch.cuda.synchronize()
            res[name] = (na.cpu().tolist(), nt.cpu().tolist(), int(r.status.item()))
        queue.put(("ok", dist.get_backend(), res))
    except Exception as e:  # reported to the test, which fails on it
        queue.put(("error", repr(e), None))
    finally:
        if dist.is_initialized():
            dist.destroy_process_group()


def test_nccl_exchange_on_one_gpu(sh):
    # the multi-GPU exchange (torch.distributed all-gathers over NCCL) on the one
    # GPU there is: a one-rank group, whose all-gathers copy each message into
    # the gathered buffer on the device; the step must match the in-process
    # exchange bit for bit, and the oracle
    import socket
    import torch.multiprocessing as mp
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    p = ctx.Process(target=_nccl_rank, args=(port, queue))
    p.start()
    p.join(300)
    if p.is_alive():  # a rendezvous that never completed
        p.kill()
        p.join()
    assert p.exitcode == 0
    kind, backend, res = queue.get(timeout=10)
    assert kind == "ok", backend
    assert backend == "nccl"
    assert res["nccl"] == res["local"]
    w = synthetic(16, 5, 32128, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.2, seed=51)
    na, nt, st = res["nccl"]
    assert_sharded_parity(w, (np.array(na), np.array(nt), st), oracle.verify_workload(w))
