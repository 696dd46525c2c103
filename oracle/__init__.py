"""TEST INFRASTRUCTURE: ctypes front end of the fp64 CPU oracle (sc_oracle.c).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` import this package.  It never imports the CUDA library or the
product package, and the product package never imports it.

Inputs are plain numpy arrays (float32 logits, or uint16 bf16 bit patterns),
as drawn by the seeded generators.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "sc_oracle.c")
LIB = os.path.join(HERE, "_build", "libscoracle.so")

RULES = {"chow": 0, "diff": 1, "opt": 2, "always": 3, "never": 4,
         "token_v1": 5, "token_v2": 6, "token_v3": 7, "lossy": 8, "bild": 9,
         "chow_log": 10, "diff_log": 11, "opt_log": 12}
DTYPES = {"f32": 0, "bf16": 1}
ROW = dict(maxq=0, maxp=1, tv=2, delta=3, accept=4, qx=5, pix=6, margin_delta=7, margin_accept=8)
SEQ = dict(min_margin=0, sample_margin=1, status=2, bonus_maxp=3)
FLAG_MARGIN = 1e-6  # decisions closer than this to flipping are not compared bit-exactly

_lib = None


def build(force: bool = False) -> str:
    """Compile sc_oracle.c with gcc (-O2, no fast-math, OpenMP)."""
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-Wall",
                    "-o", tmp, SRC, "-lm"], check=True)
    os.replace(tmp, LIB)
    return LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(LIB)
        P, I, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
        L.oracle_verify.argtypes = [P, P, I, P, P, I, I, I, I, D, D, D, P, P, P, P, I]
        L.oracle_verify.restype = I
        L.oracle_row_stats.argtypes = [P, P, I, I, I, I, D, P, P, P, I]
        L.oracle_row_stats.restype = I
        L.oracle_softmax.argtypes = [P, I, I, D, P]
        L.oracle_softmax.restype = I
        L.oracle_tv.argtypes = [P, P, I]
        L.oracle_tv.restype = D
        L.oracle_deferral.argtypes = [I, D, D, D, D, P]
        L.oracle_deferral.restype = I
        L.oracle_inverse_cdf.argtypes = [P, I, D, P]
        L.oracle_inverse_cdf.restype = I
        L.oracle_num_threads.argtypes = [I]
        L.oracle_num_threads.restype = I
        _lib = L
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _logits(a, dtype):
    want = np.uint16 if dtype == "bf16" else np.float32
    a = np.ascontiguousarray(a)
    if a.dtype != want:
        raise TypeError(f"{dtype} logits must be stored as {want.__name__}, got {a.dtype}")
    return a


def num_threads(n: int = 0) -> int:
    return lib().oracle_num_threads(n)


@dataclass
class OracleResult:
    num_accepted: np.ndarray  # [B] int32
    next_token: np.ndarray  # [B] int32
    rows: np.ndarray  # [B, gamma, 9] float64, fields in ROW
    seqs: np.ndarray  # [B, 4] float64, fields in SEQ

    @property
    def min_margin(self):
        return self.seqs[:, SEQ["min_margin"]]

    @property
    def flagged(self):
        """Sequences with a decision closer than FLAG_MARGIN to flipping."""
        return self.min_margin < FLAG_MARGIN

    @property
    def status(self):
        return self.seqs[:, SEQ["status"]].astype(np.int32)

    def row(self, name):
        return self.rows[:, :, ROW[name]]


def verify(draft, target, dtype, tokens, uniforms, B, gamma, V, rule, alpha, temperature,
           nthreads: int = 0, beta: float = 1.0) -> OracleResult:
    """GenSpecSample (Algorithm 4) with the SpecCascade target (Algorithm 5), a
    token-specific target (Section 4.4) or a Table 3 target (lossy speculative
    decoding with parameter beta, BiLD*), in fp64."""
    draft, target = _logits(draft, dtype), _logits(target, dtype)
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    uniforms = np.ascontiguousarray(uniforms, dtype=np.float32)
    assert draft.size == B * gamma * V and target.size == B * (gamma + 1) * V
    assert tokens.size == B * gamma and uniforms.size == B * (gamma + 1)
    na = np.zeros(B, np.int32)
    nt = np.zeros(B, np.int32)
    rows = np.zeros((B, gamma, len(ROW)), np.float64)
    seqs = np.zeros((B, len(SEQ)), np.float64)
    rc = lib().oracle_verify(_ptr(draft), _ptr(target), DTYPES[dtype], _ptr(tokens), _ptr(uniforms),
                             B, gamma, V, RULES[rule] if isinstance(rule, str) else int(rule),
                             float(alpha), float(beta), float(temperature), _ptr(na), _ptr(nt), _ptr(rows),
                             _ptr(seqs), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_verify rejected its arguments")
    return OracleResult(na, nt, rows, seqs)


def verify_workload(w, nthreads: int = 0, rule=None, alpha=None, beta=None) -> OracleResult:
    """``verify`` on any object with the generator's workload attributes."""
    return verify(w.draft, w.target, w.dtype, w.tokens, w.uniforms, w.B, w.gamma, w.V,
                  w.rule if rule is None else rule, w.alpha if alpha is None else alpha,
                  w.temperature, nthreads, getattr(w, "beta", 1.0) if beta is None else beta)


def row_stats(draft, target, dtype, B, gamma, V, temperature, nthreads: int = 0):
    """(max q, max p, D_TV) per pair (b, j < gamma), each [B*gamma] float64."""
    draft, target = _logits(draft, dtype), _logits(target, dtype)
    mq, mp, tv = (np.zeros(B * gamma, np.float64) for _ in range(3))
    rc = lib().oracle_row_stats(_ptr(draft), _ptr(target), DTYPES[dtype], B, gamma, V,
                                float(temperature), _ptr(mq), _ptr(mp), _ptr(tv), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_row_stats: bad arguments or an invalid row")
    return mq, mp, tv


def softmax(z, dtype, temperature):
    z = _logits(z, dtype)
    out = np.zeros(z.size, np.float64)
    if lib().oracle_softmax(_ptr(z), DTYPES[dtype], z.size, float(temperature), _ptr(out)) != 0:
        raise ValueError("not a distribution")
    return out


def tv(p, q):
    p = np.ascontiguousarray(p, np.float64)
    q = np.ascontiguousarray(q, np.float64)
    return lib().oracle_tv(_ptr(p), _ptr(q), p.size)


def deferral(rule, alpha, maxq, maxp, tv_):
    m = ctypes.c_double()
    d = lib().oracle_deferral(RULES[rule] if isinstance(rule, str) else int(rule), float(alpha),
                              float(maxq), float(maxp), float(tv_), ctypes.byref(m))
    return d, m.value


def inverse_cdf(w, u):
    w = np.ascontiguousarray(w, np.float64)
    m = ctypes.c_double()
    k = lib().oracle_inverse_cdf(_ptr(w), w.size, float(u), ctypes.byref(m))
    return k, m.value
