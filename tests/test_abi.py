"""The C-ABI library loads and exports every entry point include/sc.h declares,
and its host-only entry points behave (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sc.h")
SHARD_HEADER = os.path.join(ROOT, "include", "sc_shard.h")


@pytest.fixture(scope="module")
def so():
    import __graft_entry__ as g
    if not os.path.exists(g.LIB) or os.path.getmtime(g.LIB) < max(os.path.getmtime(s) for s in g.SOURCES):
        g.build_library()
    return ctypes.CDLL(g.LIB)


def declared_functions(headers=(HEADER, SHARD_HEADER)):
    names = []
    for h in headers:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names += re.findall(r"\b(sc_[a-z_0-9]+)\s*\(", text)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("sc_verify", "sc_row_stats", "sc_workspace_bytes", "sc_status_string", "sc_shard_pass1",
              "sc_shard_decide", "sc_shard_tv", "sc_shard_accept", "sc_shard_draw", "sc_shard_finish"):
        assert n in names


def test_every_declared_symbol_is_exported(so):
    for n in declared_functions():
        assert hasattr(so, n), n


def test_host_only_entry_points(so):
    so.sc_workspace_bytes.restype = ctypes.c_size_t
    so.sc_workspace_bytes.argtypes = [ctypes.c_int] * 3
    assert so.sc_workspace_bytes(0, 5, 10) == 0
    assert so.sc_workspace_bytes(8, 5, 256000) >= 8 * 4 + 2 * 8 * 6 * 4
    so.sc_status_string.restype = ctypes.c_char_p
    assert so.sc_status_string(0) == b"ok"
    assert so.sc_status_string(-1) == b"invalid argument"
    so.sc_max_vocab.argtypes = [ctypes.c_int]
    assert so.sc_max_vocab(1) >= 256000   # bf16 Gemma vocabulary
    assert so.sc_max_vocab(0) >= 256000   # f32 too


def test_null_pointers_are_rejected_without_a_gpu(so):
    P, I, F, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    so.sc_verify.argtypes = [P, P, I, P, P, I, I, I, I, F, F, P, P, P, S, P, P]
    rc = so.sc_verify(None, None, 1, None, None, 1, 1, 8, 0, 0.5, 1.0, None, None, None, 0, None, None)
    assert rc == -1
    rc = so.sc_verify(None, None, 1, None, None, 0, 1, 8, 0, 0.5, 1.0, None, None, None, 0, None, None)
    assert rc == -1


def test_header_is_plain_c(tmp_path):
    """include/sc.h is a C header: a C11 translation unit that calls every entry
    point compiles with warnings as errors."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    cuda_inc = next((d for d in ("/usr/local/cuda/include",) if os.path.isdir(d)), None)
    if not gcc or not cuda_inc:
        pytest.skip("gcc or the CUDA headers are missing")
    src = tmp_path / "use_sc.c"
    src.write_text("""
#include "sc.h"
int use_sc(const void *q, const void *p, const int32_t *x, const float *u, int32_t *na, int32_t *nt,
           float *mq, float *mp, float *tv, float *rows, int32_t *st, cudaStream_t s) {
  size_t n = sc_workspace_bytes(2, 3, 100);
  void *ws = 0;
  int rc = sc_workspace_init(ws, n, s);
  rc |= sc_verify(q, p, SC_BF16, x, u, 2, 3, 100, SC_RULE_OPT, 0.2f, 1.0f, na, nt, ws, n, st, s);
  rc |= sc_verify_rows(q, p, SC_F32, x, u, 2, 3, 100, SC_RULE_TOKEN_V3, 0.3f, 0.7f, na, nt, ws, n, st, rows, s);
  rc |= sc_row_stats(q, p, SC_BF16, 2, 3, 100, 1.0f, mq, mp, tv, s);
  rc |= sc_verify_static(q, p, SC_BF16, x, u, 2, 3, 100, SC_RULE_DIFF, 0.1f, 1.0f, na, nt, st, s);
  rc |= sc_verify_ex(q, p, SC_BF16, x, u, 2, 3, 100, SC_RULE_LOSSY, 0.3f, 0.9f, 1.0f, na, nt, ws, n, st, rows, s);
  rc |= sc_verify(q, p, SC_BF16, x, u, 2, 3, 100, SC_RULE_OPT_LOG, 0.5f, 0.0f, na, nt, ws, n, st, s);
  rc |= sc_debug_line(0);
  return rc + sc_max_vocab(SC_BF16) + (sc_status_string(rc) != 0);
}
""")
    r = subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-I",
                        os.path.join(ROOT, "include"), "-I", cuda_inc, str(src)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_binding_constants_mirror_the_header():
    # the Python binding passes rule codes, reads row_info fields and decodes
    # device_status bits by number: each must be the header's value
    from paper_2405_19261_gb300 import binding
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    enum = dict((k, int(v)) for k, v in re.findall(r"\b(SC_RULE_[A-Z0-9_]+)\s*=\s*(\d+)", text))
    assert enum, "no sc_rule values found"
    by_name = {"SC_RULE_" + ("ALWAYS_DEFER" if n == "always" else "NEVER_DEFER" if n == "never" else n.upper()): c
               for n, c in binding.RULES.items()}
    assert by_name == enum
    defines = dict((k, int(v)) for k, v in re.findall(r"#define\s+(SC_(?:ROW|DEV)_[A-Z_]+)\s+(\d+)u?", text))
    assert binding.ROW_FIELDS == defines["SC_ROW_FIELDS"]
    for name, idx in binding.ROW.items():
        assert idx == defines["SC_ROW_" + name.upper()], name
    assert (binding.DEV_BAD_TOKEN, binding.DEV_BAD_LOGIT, binding.DEV_BAD_UNIFORM, binding.DEV_TIMEOUT) == (
        defines["SC_DEV_BAD_TOKEN"], defines["SC_DEV_BAD_LOGIT"], defines["SC_DEV_BAD_UNIFORM"], defines["SC_DEV_TIMEOUT"])


def test_shard_host_only_entry_points(so):
    S, I = ctypes.c_size_t, ctypes.c_int
    so.sc_shard_message_bytes.restype = S
    so.sc_shard_message_bytes.argtypes = [I, I, I]
    so.sc_shard_workspace_bytes.restype = S
    so.sc_shard_workspace_bytes.argtypes = [I, I, I, I]
    B, g = 512, 8
    # message 1: (m_q, s_q, m_p, s_p) per unit, the draft token's two logits and
    # the Bhattacharyya sum per pair; 2 (OPT): a part of the lower bound on D_TV
    # per pair; 3 (OPT): a part of S_q D_TV per pair; 4: a total weight per
    # sequence; 5: a token
    assert so.sc_shard_message_bytes(B, g, 1) == B * (g + 1) * 16 + B * g * 8 + B * g * 4
    assert so.sc_shard_message_bytes(B, g, 2) == B * g * 4
    assert so.sc_shard_message_bytes(B, g, 3) == B * g * 8
    assert so.sc_shard_message_bytes(B, g, 4) == B * 8
    assert so.sc_shard_message_bytes(B, g, 5) == B * 4
    assert so.sc_shard_message_bytes(B, g, 6) == 0 and so.sc_shard_message_bytes(0, g, 1) == 0
    # independent of V: the messages are tiny against the 4.46 GB of logits
    assert sum(so.sc_shard_message_bytes(B, g, k) for k in (1, 2, 3, 4, 5)) < 200_000
    small, big = so.sc_shard_workspace_bytes(B, g, 8192, 1), so.sc_shard_workspace_bytes(B, g, 128000, 1)
    assert 0 < small < big
    assert so.sc_shard_workspace_bytes(B, g, 0, 1) == 0


def test_shard_calls_reject_bad_arguments_without_a_gpu(so):
    P, I, F, S, L64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t, ctypes.c_int64
    IA = ctypes.POINTER(ctypes.c_int)
    so.sc_shard_pass1.argtypes = [P, P, I, L64, P, I, I, I, I, IA, F, I, P, S, P, P]
    good = (ctypes.c_int * 3)(0, 100, 200)
    unordered = (ctypes.c_int * 3)(0, 150, 120)
    not_zero = (ctypes.c_int * 3)(5, 100, 200)
    for bounds, W, rank, T in ((good, 2, 0, 1.0), (good, 2, 2, 1.0), (unordered, 2, 0, 1.0),
                               (not_zero, 2, 0, 1.0), (good, 2, 0, 0.0), (good, 17, 0, 1.0), (None, 2, 0, 1.0)):
        rc = so.sc_shard_pass1(None, None, 1, 100, None, 4, 3, W, rank, bounds, T, 2, None, 0, None, None)
        assert rc == -1, (W, rank, T)
    # a batch whose grids would not fit is refused before anything else
    rc = so.sc_shard_pass1(None, None, 1, 100, None, 1 << 24, 255, 2, 0, good, 1.0, 2, None, 0, None, None)
    assert rc == -1
    so.sc_shard_finish.argtypes = [P, I, I, I, P, S, P, P, P]
    assert so.sc_shard_finish(None, 4, 3, 2, None, 0, None, None, None) == -1


def test_shard_header_is_plain_c(tmp_path):
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    cuda_inc = "/usr/local/cuda/include" if os.path.isdir("/usr/local/cuda/include") else None
    if not gcc or not cuda_inc:
        pytest.skip("gcc or the CUDA headers are missing")
    src = tmp_path / "use_shard.c"
    src.write_text("""
#include "sc_shard.h"
int use_shard(const void *q, const void *p, const int32_t *x, const float *u, void *ws, void *s1,
              void *g1, void *s2, void *g2, void *s3, void *g3, void *s4, void *g4, void *s5, void *g5,
              int32_t *na, int32_t *nt, int32_t *st, cudaStream_t s) {
  const int bounds[3] = {0, 128000, 256000};
  size_t n = sc_shard_workspace_bytes(4, 3, 128000, SC_BF16) + sc_shard_message_bytes(4, 3, 1);
  int rc = sc_shard_pass1(q, p, SC_BF16, 128000, x, 4, 3, 2, 0, bounds, 1.0f, SC_RULE_OPT, ws, n, s1, s);
  rc |= sc_shard_decide(q, p, SC_BF16, 128000, g1, x, u, 4, 3, 2, 0, bounds, SC_RULE_OPT, 0.2f, 1.0f, ws, n, s2, st, s);
  rc |= sc_shard_tv(q, p, SC_BF16, 128000, g2, 4, 3, 2, 0, bounds, SC_RULE_OPT, 0.2f, 1.0f, ws, n, s3, s);
  rc |= sc_shard_accept(q, p, SC_BF16, 128000, g3, u, 4, 3, 2, 0, bounds, SC_RULE_OPT, 0.2f, 1.0f, ws, n, s4, s);
  rc |= sc_shard_draw(q, p, SC_BF16, 128000, g4, u, 4, 3, 2, 0, bounds, 1.0f, ws, n, s5, s);
  rc |= sc_shard_finish(g5, 4, 3, 2, ws, n, na, nt, s);
  return rc + SC_SHARD_MAX;
}
""")
    r = subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-I",
                        os.path.join(ROOT, "include"), "-I", cuda_inc, str(src)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
