"""Thin ctypes binding of ``libspeccascade.so`` (include/sc.h).

Argument marshalling only: tensors are checked (device, dtype, shape,
contiguity) and their ``data_ptr()`` values are passed with the current CUDA
stream.  Every step of the verification runs in the library's kernels; a
missing library raises instead of falling back to anything else.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_lib", "libspeccascade.so")

RULES = {"chow": 0, "diff": 1, "opt": 2, "always": 3, "never": 4,
         "token_v1": 5, "token_v2": 6, "token_v3": 7, "lossy": 8, "bild": 9,
         "chow_log": 10, "diff_log": 11, "opt_log": 12}
ROW_FIELDS = 8
ROW = dict(maxq=0, maxp=1, tv=2, delta=3, accept=4, qx=5, pix=6, cand=7)
DEV_BAD_TOKEN, DEV_BAD_LOGIT, DEV_BAD_UNIFORM, DEV_TIMEOUT = 1, 2, 4, 8

_lib = None


class SCError(RuntimeError):
    pass


def lib():
    """Load the CUDA library (built by ``__graft_entry__.build()``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise SCError(f"{LIB_PATH} is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        P, I, F, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
        L.sc_workspace_bytes.argtypes = [I, I, I]
        L.sc_workspace_bytes.restype = S
        L.sc_workspace_init.argtypes = [P, S, P]
        L.sc_workspace_init.restype = I
        L.sc_max_vocab.argtypes = [I]
        L.sc_max_vocab.restype = I
        L.sc_verify.argtypes = [P, P, I, P, P, I, I, I, I, F, F, P, P, P, S, P, P]
        L.sc_verify.restype = I
        L.sc_verify_rows.argtypes = [P, P, I, P, P, I, I, I, I, F, F, P, P, P, S, P, P, P]
        L.sc_verify_rows.restype = I
        L.sc_verify_ex.argtypes = [P, P, I, P, P, I, I, I, I, F, F, F, P, P, P, S, P, P, P]
        L.sc_verify_ex.restype = I
        L.sc_row_stats.argtypes = [P, P, I, I, I, I, F, P, P, P, P]
        L.sc_row_stats.restype = I
        L.sc_debug_line.argtypes = [I]
        L.sc_debug_line.restype = I
        L.sc_status_string.argtypes = [I]
        L.sc_status_string.restype = ctypes.c_char_p
        _lib = L
    return _lib


def _check(rc: int, what: str):
    if rc != 0:
        raise SCError(f"{what}: {lib().sc_status_string(rc).decode()} ({rc})")


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return 0
    if t.dtype == torch.bfloat16:
        return 1
    raise TypeError(f"logits must be float32 or bfloat16, got {t.dtype}")


def _cuda(t: torch.Tensor, name: str, dtype=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def workspace_bytes(B: int, gamma: int, V: int = 0) -> int:
    return int(lib().sc_workspace_bytes(B, gamma, V))


def new_workspace(B: int, gamma: int, device=None) -> torch.Tensor:
    """A zeroed workspace tensor for ``sc_verify`` (reusable across calls)."""
    return torch.zeros(workspace_bytes(B, gamma), dtype=torch.uint8, device=device or "cuda")


def debug_line(reset: bool = False) -> int:
    """Kernel source line of the first failed device-side check (a library built
    with SC_DEBUG; 0: none), or -1 for a library built without the checks."""
    return int(lib().sc_debug_line(1 if reset else 0))


def max_vocab(dtype: torch.dtype) -> int:
    return int(lib().sc_max_vocab(0 if dtype == torch.float32 else 1))


def sc_verify(draft_logits: torch.Tensor, target_logits: torch.Tensor, draft_tokens: torch.Tensor,
              uniforms: torch.Tensor, rule, alpha: float, temperature: float, *,
              beta: float = 1.0,
              num_accepted: Optional[torch.Tensor] = None, next_token: Optional[torch.Tensor] = None,
              workspace: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
              row_info: Optional[torch.Tensor] = None, stream=None):
    """One verification step; returns (num_accepted [B], next_token [B]) int32.

    draft_logits [B, gamma, V], target_logits [B, gamma+1, V] (float32 or
    bfloat16, same dtype), draft_tokens [B, gamma] int32, uniforms
    [B, gamma+1] float32.  ``beta`` is lossy speculative decoding's parameter
    (rule "lossy"); temperature 0 is greedy decoding.  Outputs, workspace,
    status ([1] int32) and row_info ([B, gamma+1, 8] float32) may be passed in
    to avoid allocations.
    """
    _cuda(draft_logits, "draft_logits")
    _cuda(target_logits, "target_logits", draft_logits.dtype)
    _cuda(draft_tokens, "draft_tokens", torch.int32)
    _cuda(uniforms, "uniforms", torch.float32)
    if draft_logits.dim() != 3:
        raise ValueError("draft_logits must be [B, gamma, V]")
    B, gamma, V = draft_logits.shape
    if tuple(target_logits.shape) != (B, gamma + 1, V):
        raise ValueError(f"target_logits must be [{B}, {gamma + 1}, {V}]")
    if tuple(draft_tokens.shape) != (B, gamma) or tuple(uniforms.shape) != (B, gamma + 1):
        raise ValueError("draft_tokens must be [B, gamma] and uniforms [B, gamma+1]")
    dev = draft_logits.device
    if num_accepted is None:
        num_accepted = torch.empty(B, dtype=torch.int32, device=dev)
    if next_token is None:
        next_token = torch.empty(B, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = new_workspace(B, gamma, dev)
    for t, n in ((num_accepted, "num_accepted"), (next_token, "next_token")):
        _cuda(t, n, torch.int32)
    _cuda(workspace, "workspace")
    if status is not None:
        _cuda(status, "status", torch.int32)
    if row_info is not None:
        _cuda(row_info, "row_info", torch.float32)
        if row_info.numel() < B * (gamma + 1) * ROW_FIELDS:
            raise ValueError("row_info too small")
    rule_code = RULES[rule] if isinstance(rule, str) else int(rule)
    rc = lib().sc_verify_ex(_ptr(draft_logits), _ptr(target_logits), _dtype_code(draft_logits),
                            _ptr(draft_tokens), _ptr(uniforms), B, gamma, V, rule_code,
                            float(alpha), float(beta), float(temperature), _ptr(num_accepted),
                            _ptr(next_token), _ptr(workspace),
                            workspace.numel() * workspace.element_size(), _ptr(status),
                            _ptr(row_info), _stream(stream))
    _check(rc, "sc_verify")
    return num_accepted, next_token


def sc_row_stats(draft_logits: torch.Tensor, target_logits: torch.Tensor, temperature: float, *,
                 out=None, stream=None):
    """(max q, max p, D_TV) per pair (b, j < gamma), each [B*gamma] float32."""
    _cuda(draft_logits, "draft_logits")
    _cuda(target_logits, "target_logits", draft_logits.dtype)
    B, gamma, V = draft_logits.shape
    if tuple(target_logits.shape) != (B, gamma + 1, V):
        raise ValueError(f"target_logits must be [{B}, {gamma + 1}, {V}]")
    if out is None:
        out = tuple(torch.empty(B * gamma, dtype=torch.float32, device=draft_logits.device)
                    for _ in range(3))
    for t in out:
        _cuda(t, "row_stats output", torch.float32)
    rc = lib().sc_row_stats(_ptr(draft_logits), _ptr(target_logits), _dtype_code(draft_logits),
                            B, gamma, V, float(temperature), _ptr(out[0]), _ptr(out[1]),
                            _ptr(out[2]), _stream(stream))
    _check(rc, "sc_row_stats")
    return out


def verify(*args, **kwargs):
    """Alias of :func:`sc_verify`."""
    return sc_verify(*args, **kwargs)


def row_stats(*args, **kwargs):
    """Alias of :func:`sc_row_stats`."""
    return sc_row_stats(*args, **kwargs)


def to_device(w, device="cuda"):
    """Copy a generator workload's arrays to the device as torch tensors."""
    import numpy as np
    if w.dtype == "bf16":
        d = torch.from_numpy(np.ascontiguousarray(w.draft).view(np.int16)).view(torch.bfloat16)
        t = torch.from_numpy(np.ascontiguousarray(w.target).view(np.int16)).view(torch.bfloat16)
    else:
        d = torch.from_numpy(np.ascontiguousarray(w.draft))
        t = torch.from_numpy(np.ascontiguousarray(w.target))
    return (d.to(device), t.to(device), torch.from_numpy(np.ascontiguousarray(w.tokens)).to(device),
            torch.from_numpy(np.ascontiguousarray(w.uniforms)).to(device))


class HostVerifier:
    """sc_verify from pinned host tensors, the host-to-device copy overlapped
    with the verification: the batch is cut into ``chunks`` groups of sequences;
    group c+1 is copied on a copy stream while group c is verified on the
    calling stream (sequences are independent, so a group is verified as soon as
    its rows land).  Device buffers, the workspace and pinned output buffers are
    allocated once and reused; a call's copies wait until the previous call has
    finished reading the device buffers.

    ``v(draft, target, tokens, uniforms, rule, alpha, temperature)`` returns the
    pinned host tensors (num_accepted [B], next_token [B]), valid once the
    calling stream reaches the end of the call (e.g. after its synchronize)."""

    def __init__(self, B: int, gamma: int, V: int, dtype: torch.dtype, chunks: int = 4, device=None):
        if not (1 <= chunks <= B):
            raise ValueError("need 1 <= chunks <= B")
        dev = torch.device(device or "cuda")
        self.B, self.gamma, self.V, self.dtype = B, gamma, V, dtype
        self.d = torch.empty(B, gamma, V, dtype=dtype, device=dev)
        self.t = torch.empty(B, gamma + 1, V, dtype=dtype, device=dev)
        self.x = torch.empty(B, gamma, dtype=torch.int32, device=dev)
        self.u = torch.empty(B, gamma + 1, dtype=torch.float32, device=dev)
        self.na = torch.empty(B, dtype=torch.int32, device=dev)
        self.nt = torch.empty(B, dtype=torch.int32, device=dev)
        step = -(-B // chunks)
        self.bounds = [(b0, min(B, b0 + step)) for b0 in range(0, B, step)]
        self.ws = new_workspace(step, gamma, dev)
        self.hna = torch.empty(B, dtype=torch.int32).pin_memory()
        self.hnt = torch.empty(B, dtype=torch.int32).pin_memory()
        self.copy = torch.cuda.Stream(device=dev)
        self.landed = [torch.cuda.Event() for _ in self.bounds]
        self.done = torch.cuda.Event()
        self.done.record(torch.cuda.current_stream(dev))

    def __call__(self, draft: torch.Tensor, target: torch.Tensor, tokens: torch.Tensor, uniforms: torch.Tensor,
                 rule, alpha: float, temperature: float, *, beta: float = 1.0):
        shapes = ((draft, (self.B, self.gamma, self.V), self.dtype), (target, (self.B, self.gamma + 1, self.V), self.dtype),
                  (tokens, (self.B, self.gamma), torch.int32), (uniforms, (self.B, self.gamma + 1), torch.float32))
        for h, shape, dt in shapes:
            if h.is_cuda or tuple(h.shape) != shape or h.dtype != dt or not h.is_contiguous():
                raise ValueError(f"host inputs must be contiguous {shape} {dt} CPU tensors (pinned for overlap)")
        comp = torch.cuda.current_stream(self.d.device)
        self.copy.wait_event(self.done)  # the previous call has read the device buffers
        for (b0, b1), ev in zip(self.bounds, self.landed):
            with torch.cuda.stream(self.copy):
                self.d[b0:b1].copy_(draft[b0:b1], non_blocking=True)
                self.t[b0:b1].copy_(target[b0:b1], non_blocking=True)
                self.x[b0:b1].copy_(tokens[b0:b1], non_blocking=True)
                self.u[b0:b1].copy_(uniforms[b0:b1], non_blocking=True)
                ev.record(self.copy)
        for (b0, b1), ev in zip(self.bounds, self.landed):
            comp.wait_event(ev)
            sc_verify(self.d[b0:b1], self.t[b0:b1], self.x[b0:b1], self.u[b0:b1], rule, alpha, temperature,
                      beta=beta, num_accepted=self.na[b0:b1], next_token=self.nt[b0:b1], workspace=self.ws,
                      stream=comp)
        self.done.record(comp)
        self.hna.copy_(self.na, non_blocking=True)
        self.hnt.copy_(self.nt, non_blocking=True)
        return self.hna, self.hnt
