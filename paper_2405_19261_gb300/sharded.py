"""Vocabulary-sharded verification (include/sc_shard.h).

Each rank holds the logits of a contiguous range of tokens of every row (a
tensor-parallel LM head).  One step is five library calls per rank (six with
OPT) with an all-gather of a small message between consecutive calls; this module only
marshals arguments and moves the messages: every step of the method runs in
the library's kernels.

    ranks = [ShardRank(B, gamma, bounds, r, dtype) for r in hosted ranks]
    num_accepted, next_token = sharded_step(ranks, shards, tokens, uniforms,
                                            rule, alpha, temperature, exchange)[0]

``exchange`` gathers the hosted ranks' messages of one phase into one buffer
holding all W ranks' messages in rank order: :class:`DistExchange` (one rank
per process, ``torch.distributed.all_gather``; NCCL on GPUs) or
:class:`LocalExchange` (all W ranks hosted by one process on one device: the
messages are concatenated on the device).
"""

from __future__ import annotations

import ctypes
from typing import List, Optional, Sequence, Tuple

import torch

from . import binding

SHARD_MAX = 16
RULES = ("chow", "diff", "opt", "always", "never")

_declared = False


def lib():
    """The CUDA library with the shard entry points declared."""
    global _declared
    L = binding.lib()
    if not _declared:
        P, I, F, S, L64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t, ctypes.c_int64
        IA = ctypes.POINTER(ctypes.c_int)
        L.sc_shard_message_bytes.argtypes = [I, I, I]
        L.sc_shard_message_bytes.restype = S
        L.sc_shard_workspace_bytes.argtypes = [I, I, I, I]
        L.sc_shard_workspace_bytes.restype = S
        L.sc_shard_pass1.argtypes = [P, P, I, L64, P, I, I, I, I, IA, F, I, P, S, P, P]
        L.sc_shard_decide.argtypes = [P, P, I, L64, P, P, P, I, I, I, I, IA, I, F, F, P, S, P, P, P]
        L.sc_shard_tv.argtypes = [P, P, I, L64, P, I, I, I, I, IA, I, F, F, P, S, P, P]
        L.sc_shard_accept.argtypes = [P, P, I, L64, P, P, I, I, I, I, IA, I, F, F, P, S, P, P]
        L.sc_shard_draw.argtypes = [P, P, I, L64, P, P, I, I, I, I, IA, F, P, S, P, P]
        L.sc_shard_finish.argtypes = [P, I, I, I, P, S, P, P, P]
        for n in ("sc_shard_pass1", "sc_shard_decide", "sc_shard_tv", "sc_shard_accept", "sc_shard_draw",
                  "sc_shard_finish"):
            getattr(L, n).restype = I
        _declared = True
    return L


def shard_bounds(V: int, W: int, align: int = 8) -> List[int]:
    """W contiguous shards of nearly equal width, every inner boundary a
    multiple of ``align`` tokens (16-byte-aligned shard starts for bf16 rows of
    a multiple of 8 tokens).  Raises if some shard would be empty."""
    if not (1 <= W <= SHARD_MAX) or V < 1:
        raise ValueError(f"need 1 <= W <= {SHARD_MAX} and V >= 1")
    step = -(-V // W)
    step = -(-step // align) * align
    b = [min(r * step, V) for r in range(W)] + [V]
    if any(b[r + 1] <= b[r] for r in range(W)):
        raise ValueError(f"V={V} does not split into {W} nonempty shards of multiples of {align}")
    return b


def message_bytes(B: int, gamma: int, k: int) -> int:
    return int(lib().sc_shard_message_bytes(B, gamma, k))


def _rule_code(rule) -> int:
    code = binding.RULES[rule] if isinstance(rule, str) else int(rule)
    if code > binding.RULES["never"]:
        raise ValueError("the sharded step takes the rules of Table 1 (chow, diff, opt) and always/never")
    return code


class ShardRank:
    """The buffers of one rank: workspace, its five messages, its outputs."""

    def __init__(self, B: int, gamma: int, bounds: Sequence[int], rank: int, dtype: torch.dtype,
                 device=None):
        self.B, self.gamma, self.rank = int(B), int(gamma), int(rank)
        self.W = len(bounds) - 1
        self.bounds = list(int(v) for v in bounds)
        self._cb = (ctypes.c_int * (self.W + 1))(*self.bounds)
        self.width = self.bounds[rank + 1] - self.bounds[rank]
        self.dtype = dtype
        dev = torch.device(device or "cuda")
        L = lib()
        nws = int(L.sc_shard_workspace_bytes(B, gamma, self.width, binding._dtype_code(torch.empty(0, dtype=dtype))))
        self.workspace = torch.empty(nws, dtype=torch.uint8, device=dev)
        self.send = [None] + [torch.zeros(message_bytes(B, gamma, k), dtype=torch.uint8, device=dev)
                              for k in (1, 2, 3, 4, 5)]
        self.num_accepted = torch.empty(B, dtype=torch.int32, device=dev)
        self.next_token = torch.empty(B, dtype=torch.int32, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)

    def _shard(self, draft: torch.Tensor, target: torch.Tensor):
        """(draft, target, dtype code, ld) of this rank's logit views."""
        for t, n, rows in ((draft, "draft", self.gamma), (target, "target", self.gamma + 1)):
            if not t.is_cuda or t.dtype != self.dtype:
                raise TypeError(f"{n} shard must be a CUDA {self.dtype} tensor")
            if t.dim() != 3 or tuple(t.shape) != (self.B, rows, self.width):
                raise ValueError(f"{n} shard must be [{self.B}, {rows}, {self.width}]")
            if t.stride(2) != 1 or t.stride(0) != rows * t.stride(1):
                raise ValueError(f"{n} shard rows must be unit-stride and evenly spaced")
        if draft.stride(1) != target.stride(1):
            raise ValueError("draft and target shards must share the row stride")
        return draft, target, binding._dtype_code(draft), draft.stride(1)

    def _gathered(self, g, k):
        binding._cuda(g, f"gathered message {k}")
        if g.numel() * g.element_size() < self.W * self.send[k].numel():
            raise ValueError(f"gathered message {k} must hold the {self.W} ranks' messages")

    def pass1(self, draft, target, tokens, temperature, rule, stream=None):
        d, t, dt, ld = self._shard(draft, target)
        binding._cuda(tokens, "draft_tokens", torch.int32)
        if tuple(tokens.shape) != (self.B, self.gamma):
            raise ValueError(f"draft_tokens must be [{self.B}, {self.gamma}]")
        rc = lib().sc_shard_pass1(binding._ptr(d), binding._ptr(t), dt, ld, binding._ptr(tokens), self.B,
                                  self.gamma, self.W, self.rank, self._cb, float(temperature), _rule_code(rule),
                                  binding._ptr(self.workspace), self.workspace.numel(),
                                  binding._ptr(self.send[1]), binding._stream(stream))
        binding._check(rc, "sc_shard_pass1")
        return self.send[1]

    def decide(self, draft, target, gathered1, tokens, uniforms, rule, alpha, temperature, stream=None):
        d, t, dt, ld = self._shard(draft, target)
        binding._cuda(uniforms, "uniforms", torch.float32)
        if tuple(uniforms.shape) != (self.B, self.gamma + 1):
            raise ValueError(f"uniforms must be [{self.B}, {self.gamma + 1}]")
        self._gathered(gathered1, 1)
        rc = lib().sc_shard_decide(binding._ptr(d), binding._ptr(t), dt, ld, binding._ptr(gathered1),
                                   binding._ptr(tokens), binding._ptr(uniforms), self.B, self.gamma, self.W,
                                   self.rank, self._cb, _rule_code(rule), float(alpha), float(temperature),
                                   binding._ptr(self.workspace), self.workspace.numel(),
                                   binding._ptr(self.send[2]), binding._ptr(self.status), binding._stream(stream))
        binding._check(rc, "sc_shard_decide")
        return self.send[2]

    def tv(self, draft, target, gathered2, rule, alpha, temperature, stream=None):
        d, t, dt, ld = self._shard(draft, target)
        self._gathered(gathered2, 2)
        rc = lib().sc_shard_tv(binding._ptr(d), binding._ptr(t), dt, ld, binding._ptr(gathered2), self.B,
                               self.gamma, self.W, self.rank, self._cb, _rule_code(rule), float(alpha),
                               float(temperature), binding._ptr(self.workspace), self.workspace.numel(),
                               binding._ptr(self.send[3]), binding._stream(stream))
        binding._check(rc, "sc_shard_tv")
        return self.send[3]

    def accept(self, draft, target, gathered3, uniforms, rule, alpha, temperature, stream=None):
        d, t, dt, ld = self._shard(draft, target)
        if gathered3 is not None:
            self._gathered(gathered3, 3)
        rc = lib().sc_shard_accept(binding._ptr(d), binding._ptr(t), dt, ld, binding._ptr(gathered3),
                                   binding._ptr(uniforms), self.B, self.gamma, self.W, self.rank, self._cb,
                                   _rule_code(rule), float(alpha), float(temperature),
                                   binding._ptr(self.workspace), self.workspace.numel(),
                                   binding._ptr(self.send[4]), binding._stream(stream))
        binding._check(rc, "sc_shard_accept")
        return self.send[4]

    def draw(self, draft, target, gathered4, uniforms, temperature, stream=None):
        d, t, dt, ld = self._shard(draft, target)
        self._gathered(gathered4, 4)
        rc = lib().sc_shard_draw(binding._ptr(d), binding._ptr(t), dt, ld, binding._ptr(gathered4),
                                 binding._ptr(uniforms), self.B, self.gamma, self.W, self.rank, self._cb,
                                 float(temperature), binding._ptr(self.workspace), self.workspace.numel(),
                                 binding._ptr(self.send[5]), binding._stream(stream))
        binding._check(rc, "sc_shard_draw")
        return self.send[5]

    def finish(self, gathered5, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
        self._gathered(gathered5, 5)
        rc = lib().sc_shard_finish(binding._ptr(gathered5), self.B, self.gamma, self.W,
                                   binding._ptr(self.workspace), self.workspace.numel(),
                                   binding._ptr(self.num_accepted), binding._ptr(self.next_token),
                                   binding._stream(stream))
        binding._check(rc, "sc_shard_finish")
        return self.num_accepted, self.next_token


class LocalExchange:
    """All W ranks in one process on one device: a phase's W messages,
    concatenated in rank order into one buffer that every rank reads."""

    def __call__(self, sends: List[torch.Tensor]) -> torch.Tensor:
        return torch.cat(sends)


class DistExchange:
    """One rank per process: ``torch.distributed`` all-gather of this rank's
    message (NCCL between GPUs, gloo on CPU), in rank order."""

    def __init__(self, group=None):
        import torch.distributed as dist
        self.dist, self.group = dist, group
        self.W = dist.get_world_size(group)

    def __call__(self, sends: List[torch.Tensor]) -> torch.Tensor:
        if len(sends) != 1:
            raise ValueError("DistExchange hosts one rank per process")
        send = sends[0]
        out = torch.empty(self.W * send.numel(), dtype=send.dtype, device=send.device)
        if self.dist.get_backend(self.group) == "nccl":
            self.dist.all_gather_into_tensor(out, send, group=self.group)
        else:
            self.dist.all_gather(list(out.chunk(self.W)), send, group=self.group)
        return out


def sharded_step(ranks: List[ShardRank], shards: List[Tuple[torch.Tensor, torch.Tensor]],
                 tokens: torch.Tensor, uniforms: torch.Tensor, rule, alpha: float, temperature: float,
                 exchange, stream=None) -> List[Tuple[torch.Tensor, torch.Tensor]]:
    """One verification step of the hosted ranks; returns each hosted rank's
    (num_accepted [B], next_token [B]) int32 (identical on every rank).

    shards[i] = (draft_shard [B, gamma, width_i], target_shard [B, gamma+1,
    width_i]) of ranks[i]; tokens [B, gamma] int32 and uniforms [B, gamma+1]
    float32 are the same on every rank."""
    code = _rule_code(rule)
    opt = code == binding.RULES["opt"]
    g1 = exchange([r.pass1(d, t, tokens, temperature, code, stream) for r, (d, t) in zip(ranks, shards)])
    s2 = [r.decide(d, t, g1, tokens, uniforms, code, alpha, temperature, stream) for r, (d, t) in zip(ranks, shards)]
    g3 = None
    if opt:  # the lower bound's parts, then the D_TV parts of the pairs it did not settle
        g2 = exchange(s2)
        g3 = exchange([r.tv(d, t, g2, code, alpha, temperature, stream) for r, (d, t) in zip(ranks, shards)])
    g4 = exchange([r.accept(d, t, g3, uniforms, code, alpha, temperature, stream)
                   for r, (d, t) in zip(ranks, shards)])
    g5 = exchange([r.draw(d, t, g4, uniforms, temperature, stream) for r, (d, t) in zip(ranks, shards)])
    return [r.finish(g5, stream) for r in ranks]


def emulated_step(draft: torch.Tensor, target: torch.Tensor, tokens: torch.Tensor, uniforms: torch.Tensor,
                  rule, alpha: float, temperature: float, bounds: Sequence[int],
                  ranks: Optional[List[ShardRank]] = None, stream=None):
    """The W-rank step run by one process on one device, each rank reading its
    shard as a view of the full [B, rows, V] logits; returns (num_accepted,
    next_token, ranks) with rank 0's outputs."""
    B, gamma, V = draft.shape
    W = len(bounds) - 1
    if ranks is None:
        ranks = [ShardRank(B, gamma, bounds, r, draft.dtype, draft.device) for r in range(W)]
    shards = [(draft[:, :, bounds[r]:bounds[r + 1]], target[:, :, bounds[r]:bounds[r + 1]]) for r in range(W)]
    out = sharded_step(ranks, shards, tokens, uniforms, rule, alpha, temperature, LocalExchange(), stream)
    return out[0][0], out[0][1], ranks


class EmulatedGraph:
    """The W-rank step on one device (emulated_step) captured into a CUDA
    graph: ``replay()`` runs every rank's kernels and the on-device exchanges
    of one step with no host work between them.  The inputs are read from the
    tensors given here; refill them in place between replays."""

    def __init__(self, draft, target, tokens, uniforms, rule, alpha, temperature, bounds, warmup: int = 2):
        self.ranks = None
        side = torch.cuda.Stream(device=draft.device)
        side.wait_stream(torch.cuda.current_stream(draft.device))
        with torch.cuda.stream(side):
            for _ in range(warmup):
                _, _, self.ranks = emulated_step(draft, target, tokens, uniforms, rule, alpha, temperature, bounds,
                                                 ranks=self.ranks)
        torch.cuda.current_stream(draft.device).wait_stream(side)
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self.num_accepted, self.next_token, _ = emulated_step(draft, target, tokens, uniforms, rule, alpha,
                                                                  temperature, bounds, ranks=self.ranks)

    def replay(self):
        self.graph.replay()
        return self.num_accepted, self.next_token
