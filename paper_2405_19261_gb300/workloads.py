"""Seeded synthetic inputs for the speculative-cascade verification step.

This module only *draws* inputs: draft-model logits, target-model logits,
draft tokens and uniforms.  It holds none of the verification arithmetic
(no softmax, no deferral rule, no acceptance test, no residual), so the fp64
oracle and the CUDA path can both consume its output without sharing any of
the method's code.

Shapes follow the verification step of GenSpecSample (Algorithm 4 with the
SpecCascade target of Algorithm 5):

* ``draft``    ``[B, gamma, V]``    logits of the drafter q for the gamma drafted positions
* ``target``   ``[B, gamma+1, V]``  logits of the verifier p for positions 0..gamma
* ``tokens``   ``[B, gamma]``       int32 draft tokens x_j ~ softmax(draft_j / T)
* ``uniforms`` ``[B, gamma+1]``     float32 in [0, 1); u[b, j<gamma] drives the
  Bernoulli acceptance draw of position j, u[b, gamma] drives the single
  residual-or-bonus sample.

Logits are float32 or bf16.  bf16 arrays are stored as their uint16 bit
patterns, produced from a float32 draw by round-to-nearest-even, so every
consumer sees identical bytes.

The paper's models (T5 v1.1, Gemma 2) and datasets are not available, so the
logit distributions stand in for them (Section 5 / Appendix E fix gamma, T and
alpha ranges; the vocabulary sizes are the T5 (32128) and Gemma (256000) ones):

* ``gauss``: draft logits i.i.d. N(0, 2^2); target = draft + N(0, sigma^2).
* ``zipf``:  logit of vocabulary rank r is -1.1 ln r + N(0, 0.5^2) under a
  random per-row permutation of the vocabulary; target = draft + N(0, sigma^2).

The bonus target row (position gamma) has no draft row; it is a fresh
draft-like row plus the same kind of noise.

Draft tokens are drawn with the Gumbel-max trick, argmax_v(y_v / T + G_v) with
G_v standard Gumbel, which samples exactly from softmax(y / T) without
evaluating a softmax.
"""

from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field
from typing import Optional

import numpy as np

RULES = {"chow": 0, "diff": 1, "opt": 2, "always": 3, "never": 4,
         "token_v1": 5, "token_v2": 6, "token_v3": 7, "lossy": 8, "bild": 9,
         "chow_log": 10, "diff_log": 11, "opt_log": 12}
DTYPES = {"f32": 0, "bf16": 1}
T5_VOCAB = 32128
GEMMA_VOCAB = 256000

# Default alpha per rule for the throughput sweep (the sweep leaves alpha open).
SWEEP_ALPHA = {"chow": 0.5, "diff": 0.1, "opt": 0.2, "token_v1": 0.1, "token_v2": 0.1, "token_v3": 0.3,
               "lossy": 0.3, "always": 0.0, "never": 0.0,
               # thresholds in nats, near the medians of D(q, p), H(q) and H(q) - H(p) on
               # the sweep's rows (about 7.4, 7.1 and 0.1)
               "bild": 7.4, "chow_log": 7.1, "diff_log": 0.1, "opt_log": 0.5}
SWEEP_POINTS = [(B, g) for B in (64, 256, 512) for g in (4, 8)]


@dataclass
class Workload:
    name: str
    B: int
    gamma: int
    V: int
    dtype: str  # "f32" or "bf16"
    draft: np.ndarray  # [B, gamma, V] float32, or uint16 bf16 bits
    target: np.ndarray  # [B, gamma+1, V]
    tokens: np.ndarray  # [B, gamma] int32
    uniforms: np.ndarray  # [B, gamma+1] float32 in [0, 1)
    rule: str
    alpha: float
    temperature: float
    # Sequence b had a rejection planted at position forced[b] (-1 = none).
    forced: Optional[np.ndarray] = None
    meta: dict = field(default_factory=dict)

    @property
    def rows(self) -> int:
        return self.B * (2 * self.gamma + 1)

    @property
    def elt_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    @property
    def logit_bytes(self) -> int:
        return self.rows * self.V * self.elt_bytes

    def algorithmic_bytes(self) -> int:
        """Logits read once, plus tokens, uniforms and the two int32 outputs."""
        return (self.logit_bytes + 4 * self.B * self.gamma
                + 4 * self.B * (self.gamma + 1) + 8 * self.B)

    def subset(self, seqs) -> "Workload":
        """The same workload restricted to the sequences ``seqs`` (copies)."""
        seqs = np.asarray(seqs)
        return Workload(
            name=f"{self.name}[subset {len(seqs)}]", B=len(seqs), gamma=self.gamma,
            V=self.V, dtype=self.dtype,
            draft=np.ascontiguousarray(self.draft[seqs]),
            target=np.ascontiguousarray(self.target[seqs]),
            tokens=np.ascontiguousarray(self.tokens[seqs]),
            uniforms=np.ascontiguousarray(self.uniforms[seqs]),
            rule=self.rule, alpha=self.alpha, temperature=self.temperature,
            forced=None if self.forced is None else self.forced[seqs].copy(),
            meta=dict(self.meta))

    def with_rule(self, rule: str, alpha: float) -> "Workload":
        w = Workload(**{k: getattr(self, k) for k in self.__dataclass_fields__})
        w.rule, w.alpha = rule, float(alpha)
        w.name = f"{self.name}[{rule} a={alpha}]"
        return w


# ---------------------------------------------------------------- bit helpers

def _row_blocks(n_rows: int, row_len: int, fn, threads: bool = True) -> None:
    """fn(i0, i1) over blocks of rows, on a thread pool when the work is large
    (numpy releases the GIL inside its element-wise loops, and each element's
    result does not depend on how the rows are split).  ``threads=False`` runs
    the blocks in this thread (a caller that is itself one of a pool's tasks)."""
    per = max(1, (1 << 18) // max(1, row_len))  # ~256K elements per task
    blocks = [(i, min(n_rows, i + per)) for i in range(0, n_rows, per)]
    if not threads or len(blocks) < 2 or n_rows * row_len < (1 << 20):
        for i0, i1 in blocks:
            fn(i0, i1)
        return
    with ThreadPoolExecutor(max_workers=min(len(blocks), os.cpu_count() or 1)) as ex:
        list(ex.map(lambda bl: fn(*bl), blocks))


def f32_to_bf16_bits(x: np.ndarray, threads: bool = True) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns uint16 bits.

    Inputs must be finite (the generators only make finite values)."""
    src = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(src.shape, dtype=np.uint16)
    n = src.shape[-1] if src.ndim else 1
    b2 = src.reshape(-1, n).view(np.uint32)
    o2 = out.reshape(-1, n)

    def work(i0, i1):
        b = b2[i0:i1]
        b = b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))
        o2[i0:i1] = b >> np.uint32(16)

    _row_blocks(b2.shape[0], n, work, threads)
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def logits_as_f64(arr: np.ndarray, dtype: str) -> np.ndarray:
    """Decode stored logits (float32 or bf16 bits) to float64, exactly."""
    if dtype == "bf16":
        return bf16_bits_to_f32(arr).astype(np.float64)
    return np.asarray(arr, dtype=np.float32).astype(np.float64)


def draw_uniforms(rng: np.random.Generator, shape) -> np.ndarray:
    """float32 uniforms k * 2^-24, k uniform in [0, 2^24): always < 1."""
    k = rng.integers(0, 1 << 32, size=shape, dtype=np.uint64) >> np.uint64(8)
    return (k.astype(np.float64) * 2.0 ** -24).astype(np.float32)


def gumbel_argmax(rng: np.random.Generator, y: np.ndarray, temperature: float,
                  threads: bool = True) -> np.ndarray:
    """One exact sample per row from softmax(y / T) by the Gumbel-max trick; with
    T = 0 (greedy decoding) the row's argmax, lowest index on ties."""
    y = np.asarray(y, dtype=np.float64)
    u = rng.random(size=y.shape)
    if temperature == 0:
        return np.argmax(y, axis=-1).astype(np.int32)
    n = y.shape[-1]
    y2, u2 = y.reshape(-1, n), u.reshape(-1, n)
    out = np.empty(y2.shape[0], dtype=np.int32)

    def work(i0, i1):
        # g = -log(-log(u)), u in [0, 1) kept off 0 so that the logs stay finite
        g = np.maximum(u2[i0:i1], 1e-300)
        np.log(g, out=g)
        np.negative(g, out=g)
        np.log(g, out=g)
        np.negative(g, out=g)
        s = y2[i0:i1] / temperature
        s += g
        out[i0:i1] = np.argmax(s, axis=-1)

    _row_blocks(y2.shape[0], n, work, threads)
    return out.reshape(y.shape[:-1])


# ---------------------------------------------------------------- row draws

def _gauss_rows(rng, n, V):
    return rng.standard_normal((n, V), dtype=np.float32) * np.float32(2.0)


_ZIPF_BASE = {}


def _zipf_rows(rng, n, V):
    base = _ZIPF_BASE.get(V)
    if base is None:
        base = (-1.1 * np.log(np.arange(1, V + 1, dtype=np.float64))).astype(np.float32)
        _ZIPF_BASE[V] = base
    out = np.empty((n, V), dtype=np.float32)
    for i in range(n):
        out[i] = base[rng.permutation(V)]
    out += rng.standard_normal((n, V), dtype=np.float32) * np.float32(0.5)
    return out


def _store(x: np.ndarray, dtype: str, threads: bool = True) -> np.ndarray:
    return f32_to_bf16_bits(x, threads) if dtype == "bf16" else np.ascontiguousarray(x, dtype=np.float32)


def synthetic(B: int, gamma: int, V: int, *, dtype: str = "bf16", kind: str = "zipf",
              sigma=0.7, rule: str = "opt", alpha: float = 0.2,
              temperature: float = 1.0, seed: int = 0,
              force_reject_frac: float = 0.0, force_boost: float = 12.0,
              name: Optional[str] = None, block_rows: int = 64) -> Workload:
    """Draw one workload.

    ``sigma`` is the target-noise standard deviation: a float, or a pair
    (lo, hi) meaning sigma ~ U[lo, hi] independently per target row.
    ``force_reject_frac``: each sequence, with this probability, gets a
    planted rejection at j0 ~ U{0, 1}: one random target logit y != x_{j0} is
    set to the row's largest logit plus ``force_boost``, so p concentrates on a
    token the drafter did not pick.
    """
    if dtype not in DTYPES:
        raise ValueError(f"dtype {dtype!r}")
    if rule not in RULES:
        raise ValueError(f"rule {rule!r}")
    ss = np.random.SeedSequence(seed)
    s_logit, s_tok, s_u, s_force, s_sigma = ss.spawn(5)
    g_u, g_force, g_sigma = (np.random.default_rng(s) for s in (s_u, s_force, s_sigma))
    rows_fn = _zipf_rows if kind == "zipf" else _gauss_rows
    elt = np.uint16 if dtype == "bf16" else np.float32
    draft = np.empty((B, gamma, V), dtype=elt)
    target = np.empty((B, gamma + 1, V), dtype=elt)
    tokens = np.empty((B, gamma), dtype=np.int32)

    if isinstance(sigma, (tuple, list)):
        sig = g_sigma.uniform(sigma[0], sigma[1], size=(B, gamma + 1)).astype(np.float32)
    else:
        sig = np.full((B, gamma + 1), sigma, dtype=np.float32)
    forced = np.full(B, -1, dtype=np.int32)
    y_forced = np.zeros(B, dtype=np.int64)
    if force_reject_frac > 0:
        hit = g_force.random(B) < force_reject_frac
        j0 = g_force.integers(0, min(2, gamma), size=B)
        forced[hit] = j0[hit]
        y_forced = g_force.integers(0, max(1, V - 1), size=B)  # then shifted past x: uniform over V \ {x}

    # Sequences are drawn in blocks (bounding the float32 temporaries), each
    # block from its own child streams of the logit and token generators, so
    # the blocks run on a thread pool and the bytes do not depend on the order
    # in which they finish.
    seq_block = max(1, block_rows // (2 * gamma + 1))
    blocks = [(b0, min(B, b0 + seq_block)) for b0 in range(0, B, seq_block)]
    ss_logit, ss_tok = s_logit.spawn(len(blocks)), s_tok.spawn(len(blocks))

    def block(i):
        b0, b1 = blocks[i]
        nb = b1 - b0
        g_logit, g_tok = np.random.default_rng(ss_logit[i]), np.random.default_rng(ss_tok[i])
        d = rows_fn(g_logit, nb * (gamma + 1), V).reshape(nb, gamma + 1, V)
        noise = g_logit.standard_normal((nb, gamma + 1, V), dtype=np.float32)
        t = d + noise * sig[b0:b1, :, None]
        # Position gamma's draft-like row only seeds the bonus target row.
        dq = _store(d[:, :gamma, :], dtype, threads=False)
        draft[b0:b1] = dq
        dq64 = logits_as_f64(dq, dtype)
        tokens[b0:b1] = gumbel_argmax(g_tok, dq64.reshape(nb * gamma, V), temperature,
                                      threads=False).reshape(nb, gamma)
        for bb in range(nb):
            j0 = forced[b0 + bb]
            if j0 >= 0:
                x = tokens[b0 + bb, j0]
                y = int(y_forced[b0 + bb])
                y = y + 1 if y >= x else y
                t[bb, j0, y] = t[bb, j0].max() + np.float32(force_boost)
        target[b0:b1] = _store(t, dtype, threads=False)

    workers = min(len(blocks), os.cpu_count() or 1)
    if workers < 2 or B * (2 * gamma + 1) * V < (1 << 22):
        for i in range(len(blocks)):
            block(i)
    else:
        with ThreadPoolExecutor(max_workers=workers) as ex:
            list(ex.map(block, range(len(blocks))))

    u = draw_uniforms(g_u, (B, gamma + 1))
    return Workload(name=name or f"synthetic(B={B},g={gamma},V={V},{dtype},{kind})",
                    B=B, gamma=gamma, V=V, dtype=dtype, draft=draft, target=target,
                    tokens=tokens, uniforms=u, rule=rule, alpha=float(alpha),
                    temperature=float(temperature),
                    forced=forced if force_reject_frac > 0 else None,
                    meta=dict(kind=kind, sigma=sigma, seed=seed))


# ---------------------------------------------------------------- named configs

CONFIG_TEXT = {
    0: "B=1 gamma=4 V=32128 f32, gauss sigma=1, T=1, chow a=0.5",
    1: "B=8 gamma=5 V=32128 bf16, gauss sigma=0.5, T=1, {chow,diff,opt} x a in {0,0.1,0.3,0.5,1}",
    2: "B=32 gamma=5 V=256000 bf16, zipf sigma=0.7, T=1, opt a=0.2",
    3: "B=128 gamma=7 V=256000 bf16, zipf sigma~U[0.2,1.5] per row, T=0.7, diff a=0.1, ~half forced early rejection",
    4: "sweep B in {64,256,512} x gamma in {4,8}, V=256000 bf16, zipf sigma=0.7, T=1, chow 0.5 / diff 0.1 / opt 0.2",
}
CFG1_ALPHAS = (0.0, 0.1, 0.3, 0.5, 1.0)


def config(cfg: int, *, seed: Optional[int] = None, rule: Optional[str] = None,
           alpha: Optional[float] = None, B: Optional[int] = None,
           gamma: Optional[int] = None, temperature: Optional[float] = None) -> Workload:
    """The named workloads (seed defaults to the config id).  ``temperature``
    replaces the sweep's T = 1 (cfg 4 only; 0 is greedy decoding)."""
    s = cfg if seed is None else seed
    if cfg == 0:
        return synthetic(1, 4, T5_VOCAB, dtype="f32", kind="gauss", sigma=1.0,
                         rule=rule or "chow", alpha=0.5 if alpha is None else alpha,
                         temperature=1.0, seed=s, name="cfg0")
    if cfg == 1:
        return synthetic(8, 5, T5_VOCAB, dtype="bf16", kind="gauss", sigma=0.5,
                         rule=rule or "chow", alpha=0.5 if alpha is None else alpha,
                         temperature=1.0, seed=s, name="cfg1")
    if cfg == 2:
        return synthetic(32, 5, GEMMA_VOCAB, dtype="bf16", kind="zipf", sigma=0.7,
                         rule=rule or "opt", alpha=0.2 if alpha is None else alpha,
                         temperature=1.0, seed=s, name="cfg2")
    if cfg == 3:
        return synthetic(128, 7, GEMMA_VOCAB, dtype="bf16", kind="zipf", sigma=(0.2, 1.5),
                         rule=rule or "diff", alpha=0.1 if alpha is None else alpha,
                         temperature=0.7, seed=s, force_reject_frac=0.5, name="cfg3")
    if cfg == 4:
        B = 64 if B is None else B
        gamma = 4 if gamma is None else gamma
        rule = rule or "opt"
        if seed is None:
            s = 100 + SWEEP_POINTS.index((B, gamma)) if (B, gamma) in SWEEP_POINTS else 100
        return synthetic(B, gamma, GEMMA_VOCAB, dtype="bf16", kind="zipf", sigma=0.7,
                         rule=rule, alpha=SWEEP_ALPHA[rule] if alpha is None else alpha,
                         temperature=1.0 if temperature is None else temperature, seed=s,
                         name=f"cfg4(B={B},g={gamma},{rule})")
    raise ValueError(f"no config {cfg}")
