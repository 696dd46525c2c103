"""sc_verify_static: verification for callers that cannot allocate device memory.

Some callers of this library may not call cudaMalloc at all -- an inference
server whose device memory is handed out by its own allocator before the first
request, or code that must not trigger an allocation (and its implicit
synchronisation) in the middle of a decode step.  sc_verify_static serves them:
they pass only inputs and outputs, and the scratch the kernel needs (tickets,
per-position decision records and per-slice totals) lives in a fixed array
inside the library.

This file checks, through the C ABI, that sc_verify_static gives the same
outputs as the workspace-taking sc_verify on two calls in a row, and that a
batch beyond the fixed scratch is refused without any work being queued.  It is
collected last so that a run stopping at the first failure has run everything
else; it also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest

from paper_2405_19261_gb300.workloads import config, synthetic

pytestmark = pytest.mark.gpu

SC_ERR_SCRATCH_LIMIT = -5
STATIC_MAX_B = 2048
STATIC_MAX_UNITS = 4096


@pytest.fixture(scope="module")
def sc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2405_19261_gb300 import binding
    L = binding.lib()
    P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    L.sc_verify_static.argtypes = [P, P, I, P, P, I, I, I, I, F, F, P, P, P, P]
    L.sc_verify_static.restype = I
    return binding, L


def _static_call(binding, L, d, t, x, u, w, na, nt, status):
    import torch
    stream = torch.cuda.current_stream()
    return L.sc_verify_static(
        ctypes.c_void_p(d.data_ptr()), ctypes.c_void_p(t.data_ptr()), 1 if w.dtype == "bf16" else 0,
        ctypes.c_void_p(x.data_ptr()), ctypes.c_void_p(u.data_ptr()), w.B, w.gamma, w.V,
        binding.RULES[w.rule], float(w.alpha), float(w.temperature),
        ctypes.c_void_p(na.data_ptr()), ctypes.c_void_p(nt.data_ptr()),
        ctypes.c_void_p(status.data_ptr()), ctypes.c_void_p(stream.cuda_stream))


def test_static_scratch_matches_workspace_entry_point(sc):
    import torch
    binding, L = sc
    # two different batches back to back: the shared scratch must not carry state over
    works = [config(1, rule="opt", alpha=0.3),
             synthetic(24, 6, 32128, dtype="bf16", kind="zipf", sigma=0.8, rule="chow",
                       alpha=0.5, temperature=0.8, seed=4242)]
    for w in works:
        d, t, x, u = binding.to_device(w)
        ref_na, ref_nt = binding.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature)
        na = torch.full((w.B,), -9, dtype=torch.int32, device="cuda")
        nt = torch.full((w.B,), -9, dtype=torch.int32, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        rc = _static_call(binding, L, d, t, x, u, w, na, nt, status)
        torch.cuda.synchronize()
        assert rc == 0, L.sc_status_string(rc)
        assert int(status.item()) == 0
        # integer outputs of the same kernel on the same inputs: bit-exact, as in the parity tests
        np.testing.assert_array_equal(na.cpu().numpy(), ref_na.cpu().numpy())
        np.testing.assert_array_equal(nt.cpu().numpy(), ref_nt.cpu().numpy())
        assert np.all(na.cpu().numpy() >= 0) and np.all(nt.cpu().numpy() >= 0)


def test_static_scratch_refuses_oversized_batches(sc):
    import torch
    binding, L = sc
    # inputs of the claimed sizes (V = 8 keeps them small), so that a regressed
    # limit check would give a wrong return code, never a read past a buffer
    for B, gamma in ((STATIC_MAX_B + 1, 1), (STATIC_MAX_UNITS // 4 + 1, 3)):
        w = synthetic(B, gamma, 8, dtype="f32", kind="gauss", sigma=1.0, rule="opt", alpha=0.2, seed=5)
        d, t, x, u = binding.to_device(w)
        na = torch.zeros(w.B, dtype=torch.int32, device="cuda")
        nt = torch.zeros(w.B, dtype=torch.int32, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        rc = _static_call(binding, L, d, t, x, u, w, na, nt, status)
        torch.cuda.synchronize()
        assert rc == SC_ERR_SCRATCH_LIMIT
        assert int(status.item()) == 0
        assert int(torch.count_nonzero(na).item()) == 0 and int(torch.count_nonzero(nt).item()) == 0
