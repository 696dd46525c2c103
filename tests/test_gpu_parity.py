"""Parity of the CUDA verification step with the fp64 oracle (GPU only).

Bar: num_accepted and next_token bit-exact on every sequence the oracle does
not flag (a decision closer than 1e-6 to flipping); max q, max p, TV, q(x) and
pi(x) within 1e-5 absolute; deferral and acceptance decisions equal wherever
their own margin is at least 1e-6.
"""
import numpy as np
import pytest

import oracle
from helpers import load_golden, rows_workload
from paper_2405_19261_gb300.workloads import config, synthetic

pytestmark = pytest.mark.gpu

TOL = 1e-5


@pytest.fixture(scope="module")
def sc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2405_19261_gb300 import binding
    binding.lib()
    return binding


def run_gpu(sc, w, rows=True, rule=None, alpha=None):
    import torch
    d, t, x, u = sc.to_device(w)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ri = torch.full((w.B, w.gamma + 1, sc.ROW_FIELDS), -7.0, dtype=torch.float32, device="cuda") if rows else None
    na, nt = sc.sc_verify(d, t, x, u, w.rule if rule is None else rule,
                          w.alpha if alpha is None else alpha, w.temperature,
                          status=status, row_info=ri)
    torch.cuda.synchronize()
    return (na.cpu().numpy(), nt.cpu().numpy(), None if ri is None else ri.cpu().numpy(),
            int(status.item()))


def assert_parity(w, gpu, ref, check_rows=True):
    na, nt, ri, status = gpu
    assert status == 0
    ok = ~ref.flagged
    bad = np.nonzero(ok & ((na != ref.num_accepted) | (nt != ref.next_token)))[0]
    assert len(bad) == 0, (f"{w.name}: {len(bad)} unflagged mismatches, first b={bad[:5]}, "
                           f"gpu={na[bad[:5]]},{nt[bad[:5]]} oracle={ref.num_accepted[bad[:5]]},{ref.next_token[bad[:5]]}")
    if ri is None or not check_rows:
        return
    g = w.gamma
    R = ri[:, :g]
    np.testing.assert_allclose(R[..., 0], ref.row("maxq"), atol=TOL)
    np.testing.assert_allclose(R[..., 1], ref.row("maxp"), atol=TOL)
    np.testing.assert_allclose(ri[:, g, 1], ref.seqs[:, oracle.SEQ["bonus_maxp"]], atol=TOL)
    tv = R[..., 2]
    have = tv >= 0
    np.testing.assert_allclose(tv[have], ref.row("tv")[have], atol=TOL)
    sure_d = ref.row("margin_delta") >= oracle.FLAG_MARGIN
    np.testing.assert_array_equal(R[..., 3][sure_d], ref.row("delta")[sure_d])
    same_d = R[..., 3] == ref.row("delta")
    sure_a = sure_d & (ref.row("margin_accept") >= oracle.FLAG_MARGIN)
    np.testing.assert_array_equal(R[..., 4][sure_a], ref.row("accept")[sure_a])
    np.testing.assert_allclose(R[..., 5], ref.row("qx"), atol=TOL)
    np.testing.assert_allclose(R[..., 6][same_d], ref.row("pix")[same_d], atol=TOL)


# ----------------------------------------------------------------- hand-worked goldens

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_worked_examples(sc, dtype):
    g = load_golden("worked_examples.json")
    for ex in g["examples"]:
        for c in ex["cases"]:
            w = rows_workload(ex["q"], ex["p"], ex["tokens"], c["u"], c["rule"], c["alpha"], dtype=dtype)
            na, nt, _, status = run_gpu(sc, w)
            assert status == 0
            assert (na[0], nt[0]) == (c["num_accepted"], c["next_token"]), (ex["name"], c)


# ----------------------------------------------------------------- named configs

def test_cfg0(sc):
    w = config(0)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


@pytest.mark.parametrize("rule", ["chow", "diff", "opt"])
@pytest.mark.parametrize("alpha", [0.0, 0.1, 0.3, 0.5, 1.0])
def test_cfg1(sc, rule, alpha):
    w = config(1, rule=rule, alpha=alpha)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("rule", ["always", "opt", "diff"])
def test_many_seeds_t5_shape(sc, seed, rule):
    w = synthetic(16, 5, 32128, dtype="bf16", kind="zipf", sigma=0.7, rule=rule,
                  alpha={"always": 0.0, "opt": 0.3, "diff": 0.05}[rule], temperature=1.0,
                  seed=1000 + seed)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


# ----------------------------------------------------------------- row statistics

ROW_STATS_CASES = {
    "cfg1": lambda: config(1),
    "zipf-256k": lambda: synthetic(3, 4, 256000, dtype="bf16", kind="zipf", sigma=0.7, seed=5, temperature=0.7),
    "f32-odd": lambda: synthetic(4, 3, 10007, dtype="f32", kind="gauss", sigma=1.0, seed=6, temperature=1.3),
    # ragged vocabularies: rows of a multiple of 16 bytes stream by TMA bulk copies,
    # the others by per-thread loads
    "bf16-4097": lambda: synthetic(5, 3, 4097, dtype="bf16", kind="gauss", sigma=1.0, seed=7),
    "bf16-32127": lambda: synthetic(3, 2, 32127, dtype="bf16", kind="zipf", sigma=0.7, seed=8),
    "f32-7": lambda: synthetic(6, 3, 7, dtype="f32", kind="gauss", sigma=1.0, seed=9),
    "bf16-8200": lambda: synthetic(4, 3, 8200, dtype="bf16", kind="gauss", sigma=1.0, seed=10),
    # long drafts
    "gamma-12": lambda: synthetic(4, 12, 32128, dtype="bf16", kind="zipf", sigma=0.7, seed=11),
    "gamma-40": lambda: synthetic(2, 40, 1000, dtype="bf16", kind="zipf", sigma=1.0, seed=12),
    # the maximum vocabulary (16 CTAs x 16 chunks of 4096 logits per row)
    "max-vocab": lambda: synthetic(1, 2, 1 << 20, dtype="bf16", kind="zipf", sigma=0.7, seed=13),
    # a Gemma-vocabulary batch, every pair through the TV pass
    "gemma-B64": lambda: config(4, B=64, gamma=4),
}


@pytest.mark.parametrize("case", list(ROW_STATS_CASES))
def test_row_stats(sc, case):
    import torch
    w = ROW_STATS_CASES[case]()
    d, t, _, _ = sc.to_device(w)
    mq, mp, tv = sc.sc_row_stats(d, t, w.temperature)
    torch.cuda.synchronize()
    rq, rp, rt = oracle.row_stats(w.draft, w.target, w.dtype, w.B, w.gamma, w.V, w.temperature)
    np.testing.assert_allclose(mq.cpu().numpy(), rq, atol=TOL)
    np.testing.assert_allclose(mp.cpu().numpy(), rp, atol=TOL)
    np.testing.assert_allclose(tv.cpu().numpy(), rt, atol=TOL)


# ----------------------------------------------------------------- edge cases

@pytest.mark.parametrize("V", [1, 2, 3, 7, 8, 9, 31, 4095, 4096, 4097, 8193, 32127])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ragged_vocab(sc, V, dtype):
    w = synthetic(5, 3, V, dtype=dtype, kind="gauss", sigma=1.0, rule="always", alpha=0.0,
                  seed=V, temperature=0.9)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))
    w2 = w.with_rule("opt", 0.25)
    assert_parity(w2, run_gpu(sc, w2), oracle.verify_workload(w2))


@pytest.mark.parametrize("rule", ["always", "never"])
@pytest.mark.parametrize("gamma", [1, 2, 8, 31, 40])
def test_gamma_range(sc, gamma, rule):
    # gamma + 1 <= 32 positions report on one 64-bit ticket word; longer drafts count arrivals
    w = synthetic(3, gamma, 1000, dtype="bf16", kind="zipf", sigma=1.0, rule=rule, alpha=0.0, seed=gamma)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


def test_degenerate_rows(sc):
    B, g, V = 6, 3, 777
    w = synthetic(B, g, V, dtype="f32", kind="gauss", sigma=1.0, rule="always", alpha=0.0, seed=77)
    w.draft[0] = 0.0                 # all-equal logits: q uniform
    w.target[0] = 0.0
    w.draft[1, :, 5] = 80.0          # one huge logit: q one-hot-like
    w.target[1, :, 9] = 80.0
    w.draft[2] *= 1e4                # +-large logits, no overflow
    w.target[2] *= 1e4
    w.draft[3, :, :100] = -np.inf    # masked tokens have probability 0
    w.target[3, :, 50:150] = -np.inf
    w.tokens[3] = 200
    w.draft[4, 0, w.tokens[4, 0]] = -200.0   # the draft token's q underflows
    w.draft[5] = w.target[5, :g]     # identical rows: TV = 0, always accepted
    w.uniforms[5] = 0.999
    ref = oracle.verify_workload(w)
    gpu = run_gpu(sc, w)
    assert_parity(w, gpu, ref)
    assert gpu[0][5] == g


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("offset,T", [(0.0, 1.0), (3000.0, 0.1), (30000.0, 1.0), (-20000.0, 0.7)])
def test_acceptance_ratio_with_offset_logits(sc, dtype, offset, T):
    # A constant added to a row leaves its softmax unchanged but makes y k, the
    # row's reference and its pass-1 sum large: the ratio p(x)/q(x) must still be
    # formed to ~1e-7.  The target rows carry the offset, the draft rows none.
    # Uniforms sit 2e-6 below or above the oracle's ratio (alternately), so every
    # informative position's accept flag pins the kernel's ratio to 2e-6.
    from paper_2405_19261_gb300.workloads import f32_to_bf16_bits
    B, g, V = 16, 6, 2048
    w = synthetic(B, g, V, dtype="f32", kind="gauss", sigma=0.6, rule="always", alpha=0.0,
                  temperature=T, seed=5)
    dq = (w.draft * np.float32(T / 2)).astype(np.float32)                     # tempered N(0, 1)
    tp = (w.target * np.float32(T / 2) + np.float32(offset)).astype(np.float32)
    if dtype == "bf16":
        dq, tp = f32_to_bf16_bits(dq), f32_to_bf16_bits(tp)
    w.draft, w.target, w.dtype = dq, tp, dtype
    w.uniforms[:] = 0.5
    ratio = np.minimum(1.0, oracle.verify_workload(w).row("pix") / oracle.verify_workload(w).row("qx"))
    inform = (ratio > 1e-3) & (ratio < 1.0 - 1e-5)
    below = (np.add.outer(np.arange(B), np.arange(g)) % 2 == 0)
    u = np.where(below, ratio - 2e-6, ratio + 2e-6)
    w.uniforms[:, :g] = np.where(inform, u, 0.5).astype(np.float32)
    assert inform.sum() >= 20
    ref = oracle.verify_workload(w)
    gpu = run_gpu(sc, w)
    assert_parity(w, gpu, ref)
    acc = gpu[2][:, :g, 4]
    np.testing.assert_array_equal(acc[inform & below], 1.0)
    np.testing.assert_array_equal(acc[inform & ~below], 0.0)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("rule,alpha", [("always", 0.0), ("opt", 0.2), ("token_v3", 0.3), ("token_v1", 0.1),
                                        ("lossy", 0.3), ("lossy", 1.0)])
def test_masked_target_logit_at_the_draft_token(sc, dtype, rule, alpha):
    # p(x) = 0 < q(x): pi(x)/q(x) = 1 - delta, so a deferred draft is rejected whatever
    # its uniform (lossy speculative decoding too, alpha = 1 being the limit
    # alpha -> 1- of min(1, p/((1 - alpha) q)) = 0); with both logits masked q(x) = 0
    # and the draft is accepted
    B, g, V = 8, 3, 600
    w = synthetic(B, g, V, dtype=dtype, kind="gauss", sigma=1.0, rule=rule, alpha=alpha, seed=41)
    ninf = np.uint16(0xFF80) if dtype == "bf16" else np.float32(-np.inf)
    for b in range(B):
        for j in range(g):
            if (b + j) % 2 == 0:
                w.target[b, j, w.tokens[b, j]] = ninf
    w.draft[1, 0, w.tokens[1, 0]] = ninf
    w.target[1, 0, w.tokens[1, 0]] = ninf
    ref = oracle.verify_workload(w)
    if rule in ("always", "lossy"):
        assert np.all(ref.num_accepted[0::2] == 0)
    assert_parity(w, run_gpu(sc, w), ref)


@pytest.mark.parametrize("rule,alpha,T", [("opt", 0.3, 1.0), ("diff", 0.05, 0.7), ("token_v3", 0.3, 1.0),
                                          ("chow", 0.5, 1.0)])
def test_self_sampled_residuals_match_the_owners_pass(sc, monkeypatch, rule, alpha, T):
    # a rejected pair storing its own residual prefixes (small batches) and the
    # owner's sampling pass (large batches) sum the same weights with the same
    # code: the draws are identical, and both match the oracle
    w = synthetic(24, 6, 32128, dtype="bf16", kind="zipf", sigma=0.7, rule=rule, alpha=alpha,
                  temperature=T, seed=61, force_reject_frac=0.5)
    ref = oracle.verify_workload(w)
    out = {}
    for mode in ("0", "1"):
        monkeypatch.setenv("SC_SPEC_RES", mode)
        out[mode] = run_gpu(sc, w)
        assert_parity(w, out[mode], ref)
    np.testing.assert_array_equal(out["0"][0], out["1"][0])
    np.testing.assert_array_equal(out["0"][1], out["1"][1])
    assert np.any(ref.num_accepted < w.gamma) and np.any(ref.num_accepted == w.gamma)


@pytest.mark.parametrize("env", [{"SC_L2_HINT": "0"}, {"SC_L2_HINT": "1"}, {"SC_POS_MAJOR": "0"},
                                 {"SC_OPT_UB": "0"}, {"SC_OPT_UB": "1"}, {"SC_SPEC_RES": "0"}])
@pytest.mark.parametrize("rule,alpha", [("opt", 0.2), ("chow", 0.5), ("token_v3", 0.3)])
def test_schedule_switches_leave_the_outputs_unchanged(sc, monkeypatch, env, rule, alpha):
    # cache hints, the unit order, the upper bound on D_TV and who samples the
    # residual change how the work is scheduled, never what is computed: the
    # outputs equal the default run's bit for bit (and the oracle's)
    w = synthetic(40, 6, 256000, dtype="bf16", kind="zipf", sigma=0.7, rule=rule, alpha=alpha, seed=91,
                  force_reject_frac=0.3)
    base = run_gpu(sc, w)
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    alt = run_gpu(sc, w)
    np.testing.assert_array_equal(alt[0], base[0])
    np.testing.assert_array_equal(alt[1], base[1])
    assert_parity(w, alt, oracle.verify_workload(w))


@pytest.mark.parametrize("rule,alpha", [("token_v3", 0.0), ("token_v3", 0.3), ("token_v2", 0.05), ("token_v1", 0.05)])
def test_token_eta_screen_and_its_fallback(sc, rule, alpha):
    # eta comes from the pass-1 screen when each thread holds at most one
    # undeferred token, else from a pass over the row.  Sequences 0-1: many tied
    # largest logits spread over the row (TokenV3 falls back; for TokenV1/V2
    # max p < alpha, so nothing is deferred); 2-3: two tied largest logits in one
    # thread's vector, q = p = 1/2 there (every rule falls back); the rest are
    # ordinary rows (the screen)
    B, g, V = 12, 4, 32128
    w = synthetic(B, g, V, dtype="bf16", kind="zipf", sigma=0.7, rule=rule, alpha=alpha, seed=71)
    top = np.uint16(0x4180)  # 16.0, above every sampled logit
    for b in range(2):
        w.draft[b, :, ::97] = top
        w.target[b, :, ::89] = top
    for b in (2, 3):
        w.draft[b, :, 1000:1002] = top
        w.target[b, :, 1000:1002] = top
        w.tokens[b] = 1000 + b % 2
    ref = oracle.verify_workload(w)
    assert_parity(w, run_gpu(sc, w), ref)


def test_invalid_inputs_flagged_on_device(sc):
    w = synthetic(5, 3, 300, dtype="f32", kind="gauss", sigma=1.0, rule="opt", alpha=0.2, seed=8)
    w.tokens[1, 2] = 300
    w.draft[2, 1, 4] = np.nan
    w.target[3, 3, 0] = np.inf
    w.uniforms[4, 0] = 1.0
    na, nt, _, status = run_gpu(sc, w)
    assert status == 1 | 2 | 4
    assert np.all(na[1:] == 0) and np.all(nt[1:] == -1)
    ref = oracle.verify_workload(w)
    assert (na[0], nt[0]) == (ref.num_accepted[0], ref.next_token[0]) or ref.flagged[0]


def test_host_argument_errors(sc):
    import torch
    w = synthetic(2, 2, 64, dtype="f32", kind="gauss", seed=1)
    d, t, x, u = sc.to_device(w)
    with pytest.raises(sc.SCError):
        sc.sc_verify(d, t, x, u, "opt", 1.5, 1.0)       # alpha outside [0, 1]
    with pytest.raises(sc.SCError):
        sc.sc_verify(d, t, x, u, "opt", 0.2, -1.0)      # T < 0 (T = 0 is greedy decoding)
    with pytest.raises(sc.SCError):
        sc.sc_verify(d, t, x, u, "token_v3", 0.2, 0.0)  # greedy decoding with a token rule
    with pytest.raises(sc.SCError):
        sc.sc_verify(d, t, x, u, 13, 0.2, 1.0)          # unknown rule
    with pytest.raises(sc.SCError):
        sc.sc_verify(d, t, x, u, "opt", 0.2, 1.0, workspace=torch.zeros(4, dtype=torch.uint8, device="cuda"))
    with pytest.raises(TypeError):
        sc.sc_verify(d.cpu(), t, x, u, "opt", 0.2, 1.0)
    # empty batches, drafts and vocabularies are refused before anything is queued
    for shape in ((0, 2, 64), (2, 0, 64), (2, 2, 0)):
        B0, g0, V0 = shape
        d0 = torch.zeros((B0, g0, V0), dtype=torch.float32, device="cuda")
        t0 = torch.zeros((B0, g0 + 1, V0), dtype=torch.float32, device="cuda")
        x0 = torch.zeros((B0, g0), dtype=torch.int32, device="cuda")
        u0 = torch.zeros((B0, g0 + 1), dtype=torch.float32, device="cuda")
        with pytest.raises(sc.SCError):
            sc.sc_verify(d0, t0, x0, u0, "opt", 0.2, 1.0, workspace=torch.zeros(1 << 16, dtype=torch.uint8, device="cuda"))
    with pytest.raises(ValueError):
        sc.sc_verify(d, t[:, :2], x, u, "opt", 0.2, 1.0)


def test_repeatable_and_workspace_reuse(sc):
    import torch
    w1 = config(1, rule="opt", alpha=0.3)
    w2 = synthetic(8, 5, 32128, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.3, seed=99)
    ws = sc.new_workspace(8, 5)
    outs = []
    for w in (w1, w2, w1):
        d, t, x, u = sc.to_device(w)
        ri = torch.zeros((w.B, w.gamma + 1, 8), device="cuda")
        na, nt = sc.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature, workspace=ws, row_info=ri)
        torch.cuda.synchronize()
        outs.append((na.cpu().numpy(), nt.cpu().numpy(), ri.cpu().numpy()))
    for a, b in zip(outs[0], outs[2]):
        np.testing.assert_array_equal(a, b)   # bitwise identical on a re-run
    # tickets are left zeroed: [8][16] 8-byte slice-rank tickets, then [8] sequence
    # tickets, each region 256-byte aligned
    assert torch.count_nonzero(ws[:1024 + 256]).item() == 0
    ref2 = oracle.verify_workload(w2)
    ok = ~ref2.flagged
    np.testing.assert_array_equal(outs[1][0][ok], ref2.num_accepted[ok])
    np.testing.assert_array_equal(outs[1][1][ok], ref2.next_token[ok])


@pytest.mark.parametrize("rule,alpha", [("opt", 0.0), ("token_v3", 0.3)])
def test_cuda_graph_capture_and_replay(sc, rule, alpha):
    # a decode loop can capture the verification in a CUDA graph: after one eager
    # call (which configures the kernel), the captured launch replays on new inputs
    # copied into the same buffers, reusing one workspace, and matches the oracle
    import torch
    wl = [synthetic(8, 5, 32128, dtype="bf16", kind="zipf", sigma=0.7, rule=rule, alpha=alpha,
                    seed=s, force_reject_frac=0.5) for s in (81, 82, 83)]
    w0 = wl[0]
    d, t, x, u = sc.to_device(w0)
    na = torch.empty(w0.B, dtype=torch.int32, device="cuda")
    nt = torch.empty(w0.B, dtype=torch.int32, device="cuda")
    ws = sc.new_workspace(w0.B, w0.gamma)

    def call():
        sc.sc_verify(d, t, x, u, rule, alpha, w0.temperature, num_accepted=na, next_token=nt, workspace=ws)

    call()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        call()
    torch.cuda.synchronize()
    for w in wl + wl[:1]:
        for dst, src in zip((d, t, x, u), sc.to_device(w)):
            dst.copy_(src)
        na.fill_(-9)
        g.replay()
        torch.cuda.synchronize()
        ref = oracle.verify_workload(w)
        ok = ~ref.flagged
        assert ok.sum() >= w.B - 1
        np.testing.assert_array_equal(na.cpu().numpy()[ok], ref.num_accepted[ok])
        np.testing.assert_array_equal(nt.cpu().numpy()[ok], ref.next_token[ok])
    assert torch.count_nonzero(ws[:(8 * 16 * w0.B + 255) // 256 * 256 + 256]).item() == 0  # tickets at rest


@pytest.mark.parametrize("alpha", [0.2, 0.5, 1.0])
@pytest.mark.parametrize("ub", ["1", "0"])
def test_opt_band_settled_by_tv_bounds(sc, monkeypatch, alpha, ub):
    # Inside the OPT band (max p - alpha <= max q < max p) the kernel first bounds
    # D_TV from below by its threads' partial masses (settling delta = 0) and,
    # where it accumulates BC = sum_v sqrt(q p) (SC_OPT_UB=1; by default only for
    # the long slices of large batches), from above by sqrt(1 - BC^2) (settling
    # delta = 1); settled rows report no TV (-1).  Their decisions must still be
    # the oracle's, with the upper bound and without it.
    from paper_2405_19261_gb300.workloads import logits_as_f64
    from scipy.special import softmax
    monkeypatch.setenv("SC_OPT_UB", ub)
    w = synthetic(24, 8, 256000, dtype="bf16", kind="zipf", sigma=0.7, rule="opt", alpha=alpha,
                  temperature=1.0, seed=31)
    gpu = run_gpu(sc, w)
    ref = oracle.verify_workload(w)
    assert_parity(w, gpu, ref)
    ri = gpu[2][:, :w.gamma]
    maxq, maxp, tv = ref.row("maxq"), ref.row("maxp"), ri[..., 2]
    band = (maxq < maxp) & (maxq >= maxp - alpha)
    settled = band & (tv < 0)
    assert settled.sum() > 0, "no band row was settled by a bound"
    np.testing.assert_array_equal(ri[..., 3][settled], ref.row("delta")[settled])
    # the rows left to the TV pass report an exact D_TV
    exact = band & ~settled
    np.testing.assert_allclose(tv[exact], ref.row("tv")[exact], atol=TOL)
    # every band row whose Hellinger bound clearly decides delta = 1 was settled by
    # it (the kernel shrinks BC by 2e-4 before the bound, far past its f32 error)
    q = softmax(logits_as_f64(w.draft, "bf16"), axis=-1)
    p = softmax(logits_as_f64(w.target[:, :w.gamma], "bf16"), axis=-1)
    bc = np.minimum(1.0, np.sum(np.sqrt(q * p), axis=-1)) * (1.0 - 2e-4)
    hub = np.sqrt(np.maximum(0.0, 1.0 - bc ** 2))
    clear = band & (maxp - maxq - alpha * hub >= 1e-3)
    if ub == "1":
        np.testing.assert_array_equal(tv[clear], -1.0)
    else:  # without the upper bound these rows take the TV pass
        np.testing.assert_allclose(tv[clear], ref.row("tv")[clear], atol=TOL)
    np.testing.assert_array_equal(ri[..., 3][clear], 1.0)


# ----------------------------------------------------------------- maximum sizes

@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("rule", ["always", "opt"])
def test_max_vocab(sc, dtype, rule):
    import torch
    V = sc.max_vocab(torch.bfloat16 if dtype == "bf16" else torch.float32)   # 16 CTAs x 16 chunks
    w = synthetic(2, 2, V, dtype=dtype, kind="zipf", sigma=0.7, rule=rule, alpha=0.2,
                  temperature=1.0, seed=11)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


@pytest.mark.parametrize("rule", ["always", "never"])
def test_max_gamma(sc, rule):
    # gamma + 1 = 256 positions: the arrival-count ticket instead of the 32-bit masks
    w = synthetic(2, 255, 1000, dtype="bf16", kind="zipf", sigma=1.0, rule=rule, alpha=0.0, seed=255)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


def test_vocab_above_the_limit_is_refused(sc):
    import torch
    V = sc.max_vocab(torch.bfloat16) + 8
    w = synthetic(1, 1, V, dtype="bf16", kind="gauss", seed=3)
    d, t, x, u = sc.to_device(w)
    with pytest.raises(sc.SCError):
        sc.sc_verify(d, t, x, u, "opt", 0.2, 1.0)


# ----------------------------------------------------------------- token-specific targets

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_token_worked_examples(sc, dtype):
    g = load_golden("token_examples.json")
    for ex in g["examples"]:
        for c in ex["cases"]:
            w = rows_workload(ex["q"], ex["p"], c["tokens"], c["u"], c["rule"], c["alpha"], dtype=dtype)
            na, nt, _, status = run_gpu(sc, w)
            assert status == 0
            assert (na[0], nt[0]) == (c["num_accepted"], c["next_token"]), (ex["name"], c)


@pytest.mark.parametrize("rule,alpha", [("token_v3", 0.0), ("token_v3", 0.3), ("token_v3", 0.6),
                                        ("token_v3", 1.0), ("token_v2", 0.1), ("token_v1", 0.1)])
@pytest.mark.parametrize("seed", range(3))
def test_token_rules_t5_shape(sc, rule, alpha, seed):
    w = synthetic(16, 5, 32128, dtype="bf16", kind="zipf", sigma=0.7, rule=rule, alpha=alpha,
                  temperature=1.0, seed=2000 + seed)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


@pytest.mark.parametrize("V,dtype", [(7, "f32"), (4097, "bf16"), (10007, "f32")])
def test_token_rules_ragged_vocab(sc, V, dtype):
    w = synthetic(5, 3, V, dtype=dtype, kind="gauss", sigma=1.0, rule="token_v3", alpha=0.3,
                  temperature=0.9, seed=V)
    assert_parity(w, run_gpu(sc, w), oracle.verify_workload(w))


@pytest.mark.parametrize("chunks", [1, 3, 8])
def test_host_verifier_overlapped_copies(sc, chunks):
    # sc_verify from pinned host tensors with the copy of each group of
    # sequences overlapping the previous group's verification: the outputs are
    # sc_verify's and the oracle's, over two calls on the same buffers
    import torch
    from paper_2405_19261_gb300.workloads import synthetic
    B, g, V = 24, 5, 32128
    hv = sc.HostVerifier(B, g, V, torch.bfloat16, chunks=chunks)
    for seed in (61, 62):
        w = synthetic(B, g, V, dtype="bf16", kind="gauss", sigma=0.5, rule="opt", alpha=0.2, seed=seed)
        d, t, x, u = sc.to_device(w)
        hd, ht, hx, hu = (a.cpu().pin_memory() for a in (d, t, x, u))
        na, nt = hv(hd, ht, hx, hu, w.rule, w.alpha, w.temperature)
        torch.cuda.synchronize()
        na1, nt1 = sc.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature)
        torch.cuda.synchronize()
        assert np.array_equal(na.numpy(), na1.cpu().numpy()) and np.array_equal(nt.numpy(), nt1.cpu().numpy())
        ref = oracle.verify_workload(w)
        ok = ~ref.flagged
        assert np.array_equal(na.numpy()[ok], ref.num_accepted[ok])
        assert np.array_equal(nt.numpy()[ok], ref.next_token[ok])
