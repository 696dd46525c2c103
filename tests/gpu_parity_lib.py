"""The GPU parity check shared by the full-size tests: one call of the CUDA
verification step, and its comparison with the fp64 oracle.

Bar (north star of the parity tests): num_accepted and next_token bit-exact on
every sequence the oracle does not flag (a decision closer than 1e-6 to
flipping, or, for a decision made by an entropy or a cross entropy, closer
than ENT_MARGIN nats); max q, max p, D_TV, q(x) and pi(x) within 1e-5
absolute; deferral and acceptance decisions equal wherever their own margin is
at least that large; the finisher's candidate token at row j* equal to the
emitted token.
"""
import numpy as np

import oracle

TOL = 1e-5
ENT_MARGIN = 1e-4
ENTROPY_RULES = ("bild", "chow_log", "diff_log", "opt_log")


def run_gpu(sc, w, beta=None, workspace=None):
    """One sc_verify call through the C ABI on the workload's own rule, alpha,
    temperature (and beta), with the device status word and row diagnostics."""
    import torch
    d, t, x, u = sc.to_device(w)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ri = torch.full((w.B, w.gamma + 1, sc.ROW_FIELDS), -7.0, dtype=torch.float32, device="cuda")
    b = getattr(w, "beta", 1.0) if beta is None else beta
    na, nt = sc.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature, beta=b, status=status,
                          row_info=ri, workspace=workspace)
    torch.cuda.synchronize()
    out = na.cpu().numpy(), nt.cpu().numpy(), ri.cpu().numpy(), int(status.item())
    del d, t, x, u
    return out


def comparable(w, ref):
    """Sequences compared bit-exactly: not flagged by the oracle, and (entropy
    rules) no entropy decision closer than ENT_MARGIN at or before j*."""
    delta_margin = ENT_MARGIN if w.rule in ENTROPY_RULES else oracle.FLAG_MARGIN
    md = ref.row("margin_delta")
    reach = np.arange(w.gamma)[None, :] <= ref.num_accepted[:, None]
    return ~(ref.flagged | ((md < delta_margin) & reach).any(1)), delta_margin


def assert_parity(w, gpu, ref, min_compared=0.8):
    """Element-by-element comparison of one GPU call with the oracle; returns
    the number of sequences compared bit-exactly."""
    na, nt, ri, status = gpu
    assert status == 0, f"{w.name}: device status {status}"
    g = w.gamma
    ok, delta_margin = comparable(w, ref)
    assert ok.mean() >= min_compared, f"{w.name}: only {ok.sum()} of {w.B} sequences comparable"
    bad = np.nonzero(ok & ((na != ref.num_accepted) | (nt != ref.next_token)))[0]
    assert len(bad) == 0, (f"{w.name}: {len(bad)} unflagged mismatches, first b={bad[:5]}, "
                           f"gpu={na[bad[:5]]},{nt[bad[:5]]} oracle={ref.num_accepted[bad[:5]]},"
                           f"{ref.next_token[bad[:5]]}")
    md, ma = ref.row("margin_delta"), ref.row("margin_accept")
    R = ri[:, :g]
    np.testing.assert_allclose(R[..., 0], ref.row("maxq"), atol=TOL)
    np.testing.assert_allclose(R[..., 1], ref.row("maxp"), atol=TOL)
    np.testing.assert_allclose(ri[:, g, 1], ref.seqs[:, oracle.SEQ["bonus_maxp"]], atol=TOL)
    tv = R[..., 2]
    have = tv >= 0
    np.testing.assert_allclose(tv[have], ref.row("tv")[have], atol=TOL)
    sure_d = md >= delta_margin
    np.testing.assert_array_equal(R[..., 3][sure_d], ref.row("delta")[sure_d])
    same_d = R[..., 3] == ref.row("delta")
    sure_a = sure_d & (ma >= oracle.FLAG_MARGIN)
    np.testing.assert_array_equal(R[..., 4][sure_a], ref.row("accept")[sure_a])
    np.testing.assert_allclose(R[..., 5], ref.row("qx"), atol=TOL)
    np.testing.assert_allclose(R[..., 6][same_d], ref.row("pix")[same_d], atol=TOL)
    # the finisher marks row j* with the emitted token
    cand = ri[np.arange(w.B), np.clip(na, 0, g), 7]
    np.testing.assert_array_equal(cand[ok], nt[ok])
    return int(ok.sum())
