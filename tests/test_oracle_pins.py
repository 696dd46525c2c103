"""Pins of the fp64 oracle to what the paper and the mathematics fix.

Nothing here compares the oracle with itself: each check is against a library
routine (scipy softmax, numpy norms), a hand-worked example of the paper's
definitions (tests/golden/), a closed form (Lemma 3's rejection rate), or the
correctness property of speculative sampling (the emitted token at every
reached position is pi-distributed), established by exact enumeration over
draft tokens and over the 2^24 float32 uniform grid.
"""
import itertools

import numpy as np
import pytest

import oracle
from helpers import load_golden, np_softmax, rows_workload
from paper_2405_19261_gb300.workloads import (bf16_bits_to_f32, f32_to_bf16_bits, logits_as_f64,
                                              synthetic)

RNG = np.random.default_rng(12345)


# ----------------------------------------------------------------- step pins

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("T", [1.0, 0.7, 0.1, 2.5])
@pytest.mark.parametrize("V", [1, 2, 7, 1000, 32128])
def test_softmax_matches_scipy(dtype, T, V):
    z = (RNG.standard_normal(V) * 3).astype(np.float32)
    if dtype == "bf16":
        z = f32_to_bf16_bits(z)
    got = oracle.softmax(z, dtype, T)
    want = np_softmax(logits_as_f64(z, dtype), T)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-300)
    assert abs(got.sum() - 1.0) < 1e-13


def test_softmax_extreme_logits():
    # +-large logits must neither overflow nor lose the head; -inf means probability 0.
    z = np.array([1e4, -1e4, 9990.0, -np.inf, 0.0], np.float32)
    got = oracle.softmax(z, "f32", 1.0)
    want = np_softmax(np.where(np.isinf(z), -1e300, z.astype(np.float64)), 1.0)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-300)
    assert got[3] == 0.0
    for bad in (np.nan, np.inf):
        with pytest.raises(ValueError):
            oracle.softmax(np.array([0.0, bad], np.float32), "f32", 1.0)
    with pytest.raises(ValueError):
        oracle.softmax(np.array([-np.inf, -np.inf], np.float32), "f32", 1.0)


def test_bf16_decoding_is_exact():
    vals = np.array([1.0, -2.0, 0.15625, 3.0e38, -1.0e-30, 0.0], np.float32)
    bits = np.array([0x3F80, 0xC000, 0x3E20], np.uint16)
    np.testing.assert_array_equal(bf16_bits_to_f32(bits), [1.0, -2.0, 0.15625])
    rt = bf16_bits_to_f32(f32_to_bf16_bits(vals))
    assert np.all(np.abs(rt - vals) <= np.abs(vals) * 2.0 ** -8)
    # the oracle widens the same bits to the same doubles: a one-hot check
    z = np.array([0x3F80, 0xFF80], np.uint16)  # 1.0, -inf
    np.testing.assert_array_equal(oracle.softmax(z, "bf16", 1.0), [1.0, 0.0])


@pytest.mark.parametrize("V", [1, 3, 50, 32128])
def test_tv_is_half_l1(V):
    p = RNG.dirichlet(np.ones(V))
    q = RNG.dirichlet(np.ones(V) * 0.3)
    assert abs(oracle.tv(p, q) - 0.5 * np.abs(p - q).sum()) < 1e-13
    assert oracle.tv(p, p) == 0.0
    # disjoint supports: TV = 1
    if V >= 2:
        a = np.zeros(V); a[0] = 1
        b = np.zeros(V); b[1] = 1
        assert oracle.tv(a, b) == 1.0


def test_row_stats_match_library_routines():
    w = synthetic(3, 4, 997, dtype="bf16", kind="zipf", sigma=0.7, seed=3, temperature=0.7)
    mq, mp, tv = oracle.row_stats(w.draft, w.target, w.dtype, w.B, w.gamma, w.V, w.temperature)
    d = logits_as_f64(w.draft, "bf16")
    t = logits_as_f64(w.target, "bf16")[:, :w.gamma]
    q = np_softmax(d, w.temperature).reshape(-1, w.V)
    p = np_softmax(t, w.temperature).reshape(-1, w.V)
    np.testing.assert_allclose(mq, q.max(1), rtol=1e-12)
    np.testing.assert_allclose(mp, p.max(1), rtol=1e-12)
    np.testing.assert_allclose(tv, 0.5 * np.abs(p - q).sum(1), rtol=1e-11, atol=1e-15)


def test_deferral_table1_golden():
    g = load_golden("table1_deferral.json")
    for c in g["cases"]:
        d, m = oracle.deferral(c["rule"], c["alpha"], c["maxq"], c["maxp"], c["tv"])
        assert d == c["delta"], c


def test_inverse_cdf_brackets_u_times_total():
    for V in (1, 2, 5, 1000):
        w = RNG.exponential(size=V)
        w[RNG.random(V) < 0.3] = 0.0
        if w.sum() == 0:
            w[-1] = 1.0
        c = np.cumsum(w)
        R = c[-1]
        for u in np.concatenate([RNG.random(300), [0.0, 1 - 2 ** -24]]):
            k, margin = oracle.inverse_cdf(w, u)
            assert 0 <= k < V and w[k] > 0
            lo = c[k - 1] if k > 0 else 0.0
            if margin > 1e-12:
                assert lo <= u * R < c[k], (V, u, k)
    assert oracle.inverse_cdf(np.zeros(4), 0.5)[0] == -1


# ----------------------------------------------------------------- worked examples

def test_residual_draw_frequencies_chi_square():
    """At a certain rejection (Algorithm 4, delta = 1), the replacement token of a
    V = 4096 row pair is norm(max(0, p - q))-distributed: 40,000 seeded draws
    of u_gamma against 32 contiguous bins of equal residual mass (chi-square),
    with max(0, p - q) from numpy's fp64 softmax of the stored logits."""
    from scipy.stats import chi2
    V, N, chunk, nbins = 4096, 40000, 4000, 32
    rng = np.random.default_rng(7)
    q_log = (rng.standard_normal(V) * 2.0).astype(np.float32)
    p_log = (q_log + rng.standard_normal(V) * 1.0).astype(np.float32)
    draft = f32_to_bf16_bits(q_log[None, None, :])
    target = f32_to_bf16_bits(np.stack([p_log, p_log])[None])
    q = np_softmax(logits_as_f64(draft[0, 0], "bf16"), 1.0)
    p = np_softmax(logits_as_f64(target[0, 0], "bf16"), 1.0)
    x = int(np.argmin(p / q))                    # p(x)/q(x) far below 0.99: rejected for sure
    assert p[x] / q[x] < 0.5
    r = np.maximum(0.0, p - q)
    r /= r.sum()
    # contiguous bins in vocabulary order, each closed once it holds 1/nbins of the mass
    bounds, acc = [], 0.0
    for t in range(V):
        acc += r[t]
        if acc >= 1.0 / nbins:
            bounds.append(t)
            acc = 0.0
    bounds[-1] = V - 1
    bounds = np.array(bounds)
    nbins = len(bounds)
    cs = np.cumsum(r)
    expected = np.diff(np.concatenate([[0.0], cs[bounds]])) * N
    assert expected.min() > 50
    ks = rng.integers(0, 1 << 24, size=N)
    counts = np.zeros(len(bounds))
    for lo in range(0, N, chunk):
        n = min(chunk, N - lo)
        u = np.stack([np.full(n, 0.99, np.float32), (ks[lo:lo + n] / float(1 << 24)).astype(np.float32)], 1)
        res = oracle.verify(np.repeat(draft, n, 0), np.repeat(target, n, 0), "bf16", np.full((n, 1), x, np.int32),
                            u, n, 1, V, "always", 0.0, 1.0)
        assert np.all(res.num_accepted == 0)
        tok = res.next_token
        assert np.all(r[tok] > 0.0)
        counts += np.bincount(np.searchsorted(bounds, tok, side="left"), minlength=nbins)
    stat = float(np.sum((counts - expected) ** 2 / expected))
    assert chi2.sf(stat, nbins - 1) > 1e-3, (stat, counts, expected)


def test_worked_examples_golden():
    g = load_golden("worked_examples.json")
    for ex in g["examples"]:
        for c in ex["cases"]:
            w = rows_workload(ex["q"], ex["p"], ex["tokens"], c["u"], c["rule"], c["alpha"])
            r = oracle.verify_workload(w)
            assert (r.num_accepted[0], r.next_token[0]) == (c["num_accepted"], c["next_token"]), \
                (ex["name"], c)
            assert not r.flagged[0]


# ----------------------------------------------------------------- closed forms

def _random_workload(V, gamma, seed, rule, alpha, T=1.0, B=64):
    w = synthetic(B, gamma, V, dtype="f32", kind="gauss", sigma=1.5, rule=rule, alpha=alpha,
                  temperature=T, seed=seed)
    return w


@pytest.mark.parametrize("seed", range(4))
def test_never_defer_accepts_every_draft(seed):
    w = _random_workload(50, 5, seed, "never", 0.0)
    r = oracle.verify_workload(w)
    assert np.all(r.num_accepted == w.gamma)
    # Chow with alpha = 1 can never defer either (max q < 0 is impossible)
    r = oracle.verify_workload(w, rule="chow", alpha=1.0)
    assert np.all(r.num_accepted == w.gamma)
    assert np.all(r.row("delta") == 0)


def test_opt_and_diff_coincide_at_alpha_zero():
    w = _random_workload(40, 4, 9, "opt", 0.0, B=128)
    a = oracle.verify_workload(w)
    b = oracle.verify_workload(w, rule="diff", alpha=0.0)
    np.testing.assert_array_equal(a.num_accepted, b.num_accepted)
    np.testing.assert_array_equal(a.next_token, b.next_token)


def test_always_defer_is_speculative_decoding():
    # delta = 1 for every row: pi(x) = p(x) everywhere, acceptance min(1, p/q)
    w = _random_workload(30, 3, 5, "always", 0.0, B=256)
    r = oracle.verify_workload(w)
    assert np.all(r.row("delta") == 1)
    np.testing.assert_allclose(r.row("pix"), np.take_along_axis(
        np_softmax(logits_as_f64(w.target, "f32")[:, :w.gamma], 1.0), w.tokens[..., None], -1)[..., 0],
        rtol=1e-12)


def test_forced_rejection_is_rejected():
    w = synthetic(24, 7, 4096, dtype="bf16", kind="zipf", sigma=(0.2, 1.5), rule="diff", alpha=0.1,
                  temperature=0.7, seed=11, force_reject_frac=1.0)
    r = oracle.verify_workload(w)
    j0 = w.forced
    assert np.all(j0 >= 0)
    assert np.all(r.num_accepted <= j0)
    b = np.arange(w.B)
    assert np.all(r.row("delta")[b, j0] == 1)
    assert np.all(r.row("accept")[b, j0] == 0)


@pytest.mark.parametrize("u0", [0.0, 0.4, 0.999])
@pytest.mark.parametrize("u_gamma,token", [(0.3, 0), (0.7, 1)])
def test_masked_target_token_is_rejected_when_deferring(u0, u_gamma, token):
    # q = (1/3, 1/3, 1/3), p = (1/2, 1/2, 0), x = 2: p(x) = 0 < q(x), so with delta = 1
    # min(1, pi(x)/q(x)) = 0 and no uniform accepts (Algorithm 4's Bernoulli draw).
    # The residual max(0, p - q) = (1/6, 1/6, 0) puts u_gamma = 0.3 on token 0, 0.7 on 1.
    q = [[1 / 3, 1 / 3, 1 / 3]]
    p = [[0.5, 0.5, 0.0], [0.2, 0.3, 0.5]]
    for dtype in ("f32", "bf16"):
        w = rows_workload(q, p, [2], [u0, u_gamma], "always", 0.0, dtype=dtype)
        r = oracle.verify_workload(w)
        assert (r.num_accepted[0], r.next_token[0]) == (0, token)
        assert r.row("accept")[0, 0] == 0 and r.row("pix")[0, 0] == 0.0
        # not deferring keeps the draft: pi = q
        r = oracle.verify_workload(w, rule="never")
        assert r.num_accepted[0] == 1 and r.row("accept")[0, 0] == 1
        # a token rule defers x (r(x) = [p(x) < (1 - alpha) max p] = 1): pi(x)/q(x) = eta p(x)/q(x) = 0
        r = oracle.verify_workload(w, rule="token_v3", alpha=0.3)
        assert r.num_accepted[0] == 0 and r.row("delta")[0, 0] == 1


def test_invalid_inputs_give_defined_outputs():
    w = _random_workload(20, 3, 1, "opt", 0.2, B=5)
    w.tokens[1, 2] = 20            # out of range
    w.draft[2, 1, 4] = np.nan      # NaN logit
    w.target[3, 3, 0] = np.inf     # +inf in the bonus row
    w.uniforms[4, 0] = 1.0         # uniform outside [0, 1)
    r = oracle.verify_workload(w)
    assert list(r.status) == [0, 1, 2, 2, 4]
    assert np.all(r.num_accepted[1:] == 0) and np.all(r.next_token[1:] == -1)
    assert r.next_token[0] >= 0


# ----------------------------------------------------------------- exact enumeration

GRID = 1 << 24  # uniforms are k * 2^-24


def _batched(w, X, K):
    """Oracle outputs for sequences that share w's rows, with draft tokens X
    [N, gamma] and uniform grid indices K [N, gamma+1]."""
    N = X.shape[0]
    draft = np.broadcast_to(w.draft[:1], (N,) + w.draft.shape[1:]).copy()
    target = np.broadcast_to(w.target[:1], (N,) + w.target.shape[1:]).copy()
    u = (K.astype(np.float64) / GRID).astype(np.float32)
    r = oracle.verify(draft, target, w.dtype, X.astype(np.int32), u, N, w.gamma, w.V, w.rule,
                      w.alpha, w.temperature, nthreads=1, beta=getattr(w, "beta", 1.0))
    return r


def _first_true(pred, N):
    """Smallest k in [0, GRID] with pred(k) true, for monotone predicates (batched)."""
    lo = np.zeros(N, np.int64)
    hi = np.full(N, GRID, np.int64)
    while np.any(lo < hi):
        mid = (lo + hi) // 2
        t = pred(np.minimum(mid, GRID - 1)) | (mid >= GRID)
        hi = np.where(t, mid, hi)
        lo = np.where(t, lo, mid + 1)
    return lo


def exact_output_law(w):
    """Exact law of the oracle's output over draft tokens x ~ prod_j q_j and the
    float32 uniform grid.  Returns per position j: P(reach j), the law of the
    token emitted at j given reach, and P(reject at j | reach j)."""
    g, V = w.gamma, w.V
    X = np.array(list(itertools.product(range(V), repeat=g)), np.int64)
    N = len(X)
    q = np_softmax(logits_as_f64(w.draft[0], w.dtype), w.temperature)
    wx = np.prod(q[np.arange(g)[None, :], X], axis=1)

    # acceptance measure a_j(x): earlier positions accept (u = 0), later ones are irrelevant
    acc = np.zeros((N, g))
    for j in range(g):
        def rejects(k, j=j):
            K = np.zeros((N, g + 1), np.int64)
            K[:, j] = k
            return _batched(w, X, K).num_accepted == j
        acc[:, j] = _first_true(rejects, N) / GRID

    def token_law(j_reject):
        # law of the sampled token as a function of u_gamma, given the acceptance pattern
        NV = N * (V + 1)
        Xr = np.repeat(X, V + 1, axis=0)
        vv = np.tile(np.arange(V + 1), N)
        base = np.zeros((NV, g + 1), np.int64)
        if j_reject < g:
            base[:, j_reject] = GRID - 1

        def at_least(k):
            K = base.copy()
            K[:, g] = k
            return _batched(w, Xr, K).next_token >= vv
        first = _first_true(at_least, NV).reshape(N, V + 1)
        first[:, V] = GRID
        first[:, 0] = 0
        return np.diff(first, axis=1) / GRID  # [N, V]

    laws, reach, reject = [], [], []
    pre = np.ones(N)
    for j in range(g + 1):
        pr = float(np.sum(wx * pre))
        if j < g:
            res = token_law(j)
            emit = acc[:, j:j + 1] * (np.arange(V)[None, :] == X[:, j:j + 1]) + (1 - acc[:, j:j + 1]) * res
            rj = float(np.sum(wx * pre * (1 - acc[:, j]))) / pr
        else:
            emit = token_law(g)
            rj = 1.0
        laws.append(np.sum((wx * pre)[:, None] * emit, axis=0) / pr)
        reach.append(pr)
        reject.append(rj)
        if j < g:
            pre = pre * acc[:, j]
    return reach, laws, reject


ENUM_CASES = [
    # (V, gamma, rule, alpha, T, seed)
    (2, 1, "always", 0.0, 1.0, 0),
    (3, 2, "always", 0.0, 1.0, 1),
    (4, 3, "always", 0.0, 0.7, 2),
    (8, 2, "always", 0.0, 1.0, 3),
    (5, 2, "never", 0.0, 1.0, 4),
    (4, 3, "chow", 0.45, 1.0, 5),
    (6, 2, "diff", 0.05, 1.0, 6),
    (4, 3, "opt", 0.3, 1.0, 7),
    (7, 2, "opt", 0.8, 0.5, 8),
    (3, 3, "diff", 0.0, 2.0, 9),
]


@pytest.mark.parametrize("V,gamma,rule,alpha,T,seed", ENUM_CASES)
def test_enumeration_emitted_token_is_pi_distributed(V, gamma, rule, alpha, T, seed):
    """Speculative sampling with a general target (Algorithm 4): conditional on
    reaching position j, the emitted token is pi_j-distributed, with
    pi_j = (1 - delta_j) q_j + delta_j p_j (Eq. 6) and pi_gamma = p_gamma; the
    rejection probability at j is delta_j * D_TV(p_j, q_j) (Lemma 3)."""
    rng = np.random.default_rng(seed)
    q_log = (rng.standard_normal((gamma, V)) * 1.5).astype(np.float32)
    p_log = (q_log[np.r_[0:gamma, gamma - 1]] + rng.standard_normal((gamma + 1, V)) * 1.2).astype(np.float32)
    w = rows_workload(np.exp(q_log), np.exp(p_log), np.zeros(gamma), np.zeros(gamma + 1), rule,
                      alpha, temperature=T)
    # rows_workload multiplies the log-probabilities by T, so softmax(z/T) = the rows above
    info = oracle.verify_workload(w)
    q = np_softmax(logits_as_f64(w.draft[0], "f32"), T)
    p = np_softmax(logits_as_f64(w.target[0], "f32"), T)
    delta = info.row("delta")[0]
    np.testing.assert_allclose(info.row("maxq")[0], q.max(1), rtol=1e-12)
    np.testing.assert_allclose(info.row("maxp")[0], p[:gamma].max(1), rtol=1e-12)
    tv = 0.5 * np.abs(p[:gamma] - q).sum(1)
    np.testing.assert_allclose(info.row("tv")[0], tv, rtol=1e-11, atol=1e-15)
    for j in range(gamma):
        assert delta[j] == oracle.deferral(rule, alpha, q[j].max(), p[j].max(), tv[j])[0]
    if rule == "always":
        assert np.all(delta == 1)
    if rule == "never":
        assert np.all(delta == 0)

    reach, laws, reject = exact_output_law(w)
    tol = 4.0 * V / GRID + 1e-9
    for j in range(gamma):
        pi = (1 - delta[j]) * q[j] + delta[j] * p[j]
        np.testing.assert_allclose(laws[j], pi, atol=tol, err_msg=f"position {j}")
        assert abs(reject[j] - delta[j] * tv[j]) < tol, (j, reject[j], delta[j] * tv[j])
    np.testing.assert_allclose(laws[gamma], p[gamma], atol=tol, err_msg="bonus position")
    # P(reach j + 1) = P(reach j) (1 - delta_j TV_j)
    for j in range(gamma):
        assert abs(reach[j + 1] - reach[j] * (1 - delta[j] * tv[j])) < tol


def _entropy_delta(rule, alpha, q, p, tv):
    """delta of BiLD* and the log-loss rules from scipy's entropies."""
    from scipy.stats import entropy
    Hq, Hp = entropy(q), entropy(p)
    if rule == "bild":
        return float(Hq + entropy(q, p) > alpha)   # D(q, p) = H(q) + KL(q || p)
    if rule == "chow_log":
        return float(Hq > alpha)
    if rule == "diff_log":
        return float(-Hq < -Hp - alpha)
    return float(-Hq < -Hp - alpha * tv)             # opt_log


TABLE3_ENUM_CASES = [
    # (V, gamma, rule, alpha, beta, T, seed); alpha None: the median of the rule's statistic
    (4, 2, "lossy", 0.3, 1.0, 1.0, 21),
    (5, 2, "lossy", 0.5, 0.6, 1.0, 22),
    (3, 3, "lossy", 0.2, 0.9, 0.7, 23),
    (4, 3, "bild", None, 1.0, 1.0, 24),
    (5, 2, "chow_log", None, 1.0, 1.0, 25),
    (4, 3, "diff_log", None, 1.0, 0.8, 26),
    (6, 2, "opt_log", 0.5, 1.0, 1.0, 27),    # position 0: the alpha D_TV term decides (DiffLog would not defer)
]


@pytest.mark.parametrize("V,gamma,rule,alpha,beta,T,seed", TABLE3_ENUM_CASES)
def test_enumeration_table3_and_log_loss_targets(V, gamma, rule, alpha, beta, T, seed):
    """Algorithm 4 with any target pi: a draft x is kept with probability
    min(1, pi(x)/q(x)) and otherwise replaced from norm(max(0, pi - q)), so the
    token emitted at a reached position has law
        min(q, pi) + (sum max(0, q - pi) / sum max(0, pi - q)) max(0, pi - q),
    which is pi itself when pi sums to one, and the rejection probability is
    sum max(0, q - pi).  pi is built here from its definition: the lossy target
    of Table 3, or (1 - delta) q + delta p with delta from scipy's entropies."""
    rng = np.random.default_rng(seed)
    q_log = (rng.standard_normal((gamma, V)) * 1.5).astype(np.float32)
    p_log = (q_log[np.r_[0:gamma, gamma - 1]] + rng.standard_normal((gamma + 1, V)) * 1.2).astype(np.float32)
    qs = np_softmax(q_log.astype(np.float64), 1.0)
    ps = np_softmax(p_log.astype(np.float64), 1.0)
    tv = 0.5 * np.abs(ps[:gamma] - qs).sum(1)
    if alpha is None:   # a threshold between the rows' statistics, so that delta takes both values
        from scipy.stats import entropy
        Hq = np.array([entropy(qs[j]) for j in range(gamma)])
        Hp = np.array([entropy(ps[j]) for j in range(gamma)])
        stat = {"bild": Hq + np.array([entropy(qs[j], ps[j]) for j in range(gamma)]),
                "chow_log": Hq, "diff_log": Hq - Hp, "opt_log": (Hq - Hp) / np.maximum(tv, 1e-3)}[rule]
        alpha = float(max(0.0, np.median(stat)))
    w = rows_workload(np.exp(q_log), np.exp(p_log), np.zeros(gamma), np.zeros(gamma + 1), rule,
                      alpha, temperature=T)
    w.beta = beta
    q = np_softmax(logits_as_f64(w.draft[0], "f32"), T)
    p = np_softmax(logits_as_f64(w.target[0], "f32"), T)
    reach, laws, reject = exact_output_law(w)
    tol = 4.0 * V / GRID + 1e-9
    for j in range(gamma):
        if rule == "lossy":
            pi = np.maximum(np.minimum(q[j], p[j] / (1.0 - alpha)), p[j] / beta)
        else:
            d = _entropy_delta(rule, alpha, q[j], p[j], 0.5 * np.abs(p[j] - q[j]).sum())
            pi = (1 - d) * q[j] + d * p[j]
        out, res = np.maximum(0.0, q[j] - pi), np.maximum(0.0, pi - q[j])
        law = np.minimum(q[j], pi) + (out.sum() / res.sum() if res.sum() > 0 else 0.0) * res
        np.testing.assert_allclose(laws[j], law, atol=tol, err_msg=f"{rule} position {j}")
        assert abs(reject[j] - out.sum()) < tol, (j, reject[j], out.sum())
        assert abs(reach[j + 1] - reach[j] * (1 - out.sum())) < tol
    np.testing.assert_allclose(laws[gamma], p[gamma], atol=tol, err_msg="bonus position")


def test_enumeration_agrees_with_fine_grid_bruteforce():
    """V = 2, gamma = 1: tally the oracle over an explicit grid of uniforms and
    draft tokens, independent of the bisection machinery above."""
    w = rows_workload([[0.7, 0.3]], [[0.2, 0.8], [0.6, 0.4]], [0], [0, 0], "always", 0.0)
    n = 512
    grid = (np.arange(n) + 0.5) / n
    q = np.array([0.7, 0.3])
    emit0 = np.zeros(2)
    for x in (0, 1):
        U = np.array(list(itertools.product(grid, grid)), np.float32)
        X = np.full((len(U), 1), x, np.int64)
        draft = np.broadcast_to(w.draft[:1], (len(U), 1, 2)).copy()
        target = np.broadcast_to(w.target[:1], (len(U), 2, 2)).copy()
        r = oracle.verify(draft, target, "f32", X.astype(np.int32), U, len(U), 1, 2, "always", 0.0, 1.0)
        tok0 = np.where(r.num_accepted >= 1, x, r.next_token)
        emit0 += q[x] * np.bincount(tok0, minlength=2) / len(U)
    np.testing.assert_allclose(emit0, [0.2, 0.8], atol=2.0 / n)


# ----------------------------------------------------------------- token-specific targets

def test_token_worked_examples():
    """Hand-worked TokenSpecCascade runs (Section 4.4) on a 4-token vocabulary."""
    g = load_golden("token_examples.json")
    for ex in g["examples"]:
        for c in ex["cases"]:
            w = rows_workload(ex["q"], ex["p"], c["tokens"], c["u"], c["rule"], c["alpha"])
            r = oracle.verify_workload(w)
            assert not r.flagged[0], (ex["name"], c)
            assert (r.num_accepted[0], r.next_token[0]) == (c["num_accepted"], c["next_token"]), (ex["name"], c)


def test_table3_and_log_loss_worked_examples():
    """Hand-worked runs of Algorithm 4 with the lossy target (Table 3, Lemma 2),
    BiLD*, the log-loss rules and greedy decoding on a 3-token vocabulary."""
    g = load_golden("table3_logloss_examples.json")
    for ex in g["examples"]:
        for c in ex["cases"]:
            # logits are the log-probabilities at T = 1; T = 0 reads the same logits greedily
            w = rows_workload(ex["q"], ex["p"], c["tokens"], c["u"], c["rule"], c["alpha"])
            w.temperature = c["T"]
            r = oracle.verify_workload(w, beta=c.get("beta", 1.0))
            assert not r.flagged[0], (ex["name"], c)
            assert (r.num_accepted[0], r.next_token[0]) == (c["num_accepted"], c["next_token"]), (ex["name"], c)


@pytest.mark.parametrize("rule", ["token_v1", "token_v2"])
def test_token_margin_counts_the_draft_token_however_light(rule):
    """The draft token's own deferral r(x) decides whether it is kept outright
    (Section 4.4: the acceptance ratio is (1 - r(x)) + eta p(x)/q(x)), so its
    comparison counts towards the sequence's decision margin even when q(x) and
    p(x) are far below the 1e-9 that lighter non-draft tokens need.  Hand-built
    row: q = (0.6, 0.4 - 5e-10, 5e-10), p = (0.5, 0.5 - 1e-10, 1e-10), and alpha
    put 6e-10 below max p, so the threshold max p - alpha = 6e-10 sits 1e-10 above
    q(2) (TokenV1) and 5e-10 above p(2) (TokenV2): r(2) = 1 with a margin far below
    1e-6.  With x = 2 the sequence is flagged; with x = 0 (r(0) = 0, margin 0.1 or
    more) the same light token does not flag it."""
    qrow = [[0.6, 0.4 - 5e-10, 5e-10]]
    prow = [[0.5, 0.5 - 1e-10, 1e-10], [0.2, 0.3, 0.5]]
    for x, flagged in ((2, True), (0, False)):
        w = rows_workload(qrow, prow, [x], [0.5, 0.37], rule, 0.4)
        maxp = oracle.verify_workload(w).row("maxp")[0, 0]
        w.alpha = float(maxp - 6e-10)
        r = oracle.verify_workload(w)
        q = np_softmax(logits_as_f64(w.draft[0, 0], "f32"), 1.0)
        p = np_softmax(logits_as_f64(w.target[0, 0], "f32"), 1.0)
        light = q[2] if rule == "token_v1" else p[2]
        assert light < 1e-9 and abs(light - 6e-10) < 6e-10
        if flagged:
            assert r.row("delta")[0, 0] == 1            # r(x) = 1: the light draft is deferred
            assert abs(r.row("margin_delta")[0, 0] - abs(light - 6e-10)) < 1e-15
            assert r.flagged[0]
        else:
            assert r.row("delta")[0, 0] == 0 and r.num_accepted[0] == 1
            assert r.row("margin_delta")[0, 0] > 0.09
            assert not r.flagged[0]


def _token_pi(rule, alpha, q, p):
    """pi_Token(v) = q(v)(1 - r(v)) + eta p(v), eta = sum_v r(v) q(v), for one row
    (Section 4.4; r by the TokenV1 / TokenV2 / TokenV3 plug-in rules)."""
    maxp = p.max()
    if rule == "token_v1":
        r = q < maxp - alpha
    elif rule == "token_v2":
        r = p < maxp - alpha
    else:
        r = p < maxp * (1.0 - alpha)
    eta = q[r].sum()
    return np.where(r, 0.0, q) + eta * p, r


TOKEN_ENUM_CASES = [
    # (V, gamma, rule, alpha, T, seed)
    (4, 2, "token_v3", 0.3, 1.0, 21),
    (5, 2, "token_v3", 0.6, 0.8, 22),
    (6, 1, "token_v3", 0.0, 1.0, 23),
    (4, 3, "token_v2", 0.1, 1.0, 24),
    (5, 2, "token_v1", 0.2, 1.0, 25),
    (3, 3, "token_v1", 0.05, 1.5, 26),
]


@pytest.mark.parametrize("V,gamma,rule,alpha,T,seed", TOKEN_ENUM_CASES)
def test_enumeration_token_specific_target(V, gamma, rule, alpha, T, seed):
    """Speculative sampling with the token-specific target: conditional on
    reaching position j, the emitted token is pi_Token-distributed, pi_Token sums
    to one, and the rejection probability at j is sum_v max(0, q(v) - pi(v))
    (Lemma 3 with pi in place of p); the bonus token is p_gamma-distributed."""
    rng = np.random.default_rng(seed)
    q_log = (rng.standard_normal((gamma, V)) * 1.5).astype(np.float32)
    p_log = (q_log[np.r_[0:gamma, gamma - 1]] + rng.standard_normal((gamma + 1, V)) * 1.2).astype(np.float32)
    w = rows_workload(np.exp(q_log), np.exp(p_log), np.zeros(gamma), np.zeros(gamma + 1), rule,
                      alpha, temperature=T)
    info = oracle.verify_workload(w)
    q = np_softmax(logits_as_f64(w.draft[0], "f32"), T)
    p = np_softmax(logits_as_f64(w.target[0], "f32"), T)
    reach, laws, reject = exact_output_law(w)
    tol = 4.0 * V / GRID + 1e-9
    for j in range(gamma):
        pi, r = _token_pi(rule, alpha, q[j], p[j])
        assert abs(pi.sum() - 1.0) < 1e-12
        assert info.row("delta")[0][j] == r[0]   # reported: r(x_j), x_j = 0 in the stored tokens
        np.testing.assert_allclose(laws[j], pi, atol=tol, err_msg=f"position {j}")
        assert abs(reject[j] - np.maximum(0.0, q[j] - pi).sum()) < tol, (j, reject[j])
    np.testing.assert_allclose(laws[gamma], p[gamma], atol=tol, err_msg="bonus position")


@pytest.mark.parametrize("rule", ["token_v1", "token_v2", "token_v3"])
def test_token_rules_that_defer_nothing_accept_every_draft(rule):
    # alpha = 1: TokenV3 compares p(v) < 0 and TokenV1/V2 compare with max p - 1 <= 0,
    # so r = 0 everywhere, eta = 0 and pi = q: every draft is accepted
    w = synthetic(8, 5, 1000, dtype="bf16", kind="zipf", sigma=1.0, rule=rule, alpha=1.0, seed=41)
    r = oracle.verify_workload(w)
    assert np.all(r.num_accepted == w.gamma)
    assert np.all(r.row("delta") == 0) and np.all(r.row("accept") == 1)
    np.testing.assert_allclose(r.row("pix"), r.row("qx"), rtol=1e-12)


# ----------------------------------------------------------------- Table 3 targets

def _lossy_sd_direct(q, p, x, u, alpha, beta):
    """Lossy speculative decoding as its own procedure (Section 2): accept x_j with
    probability min(1, p(x)/((1 - alpha) q(x))); at the first rejection draw from
    norm(max(0, p/beta - q)); after full acceptance draw from p_gamma.  Inverse
    CDF in ascending vocabulary order with the last uniform."""
    g = len(x)
    for j in range(g):
        rho = min(1.0, p[j][x[j]] / ((1.0 - alpha) * q[j][x[j]])) if alpha < 1 else 1.0
        if not u[j] < rho:
            wts = np.maximum(0.0, p[j] / beta - q[j])
            c = np.cumsum(wts)
            return j, int(np.searchsorted(c, u[g] * c[-1], side="right")), abs(u[j] - rho)
    c = np.cumsum(p[g])
    return g, int(np.searchsorted(c, u[g] * c[-1], side="right")), np.inf


@pytest.mark.parametrize("alpha,beta", [(0.0, 1.0), (0.2, 1.0), (0.5, 0.5), (0.5, 1.3), (0.9, 0.4)])
@pytest.mark.parametrize("seed", range(3))
def test_lossy_target_reproduces_lossy_speculative_decoding(alpha, beta, seed):
    """Lemma 2: Algorithm 4 with pi = max{min{q, p/(1 - alpha)}, p/beta} accepts and
    resamples exactly as lossy speculative decoding does."""
    rng = np.random.default_rng(300 + seed)
    V, g = 6, 2
    q_log = (rng.standard_normal((g, V)) * 1.5).astype(np.float32)
    p_log = (q_log[np.r_[0:g, g - 1]] + rng.standard_normal((g + 1, V))).astype(np.float32)
    q = np_softmax(q_log.astype(np.float64), 1.0)
    p = np_softmax(p_log.astype(np.float64), 1.0)
    checked = 0
    for trial in range(60):
        x = rng.integers(0, V, size=g)
        u = rng.random(g + 1).astype(np.float32)
        w = rows_workload(np.exp(q_log), np.exp(p_log), x, u, "lossy", alpha)
        w.beta = beta
        r = oracle.verify_workload(w)
        qq = np_softmax(logits_as_f64(w.draft[0], "f32"), 1.0)
        pp = np_softmax(logits_as_f64(w.target[0], "f32"), 1.0)
        ja, tok, margin = _lossy_sd_direct(qq, pp, x, u.astype(np.float64), alpha, beta)
        if margin < 1e-9 or r.flagged[0]:
            continue
        assert (r.num_accepted[0], r.next_token[0]) == (ja, tok), (trial, x, u)
        checked += 1
    assert checked > 40


def test_lossy_at_alpha_0_beta_1_is_standard_speculative_sampling():
    # alpha = 0, beta = 1: pi = max{min{q, p}, p} = p, Algorithm 1
    w = synthetic(16, 5, 2000, dtype="bf16", kind="zipf", sigma=0.7, rule="lossy", alpha=0.0, seed=51)
    a = oracle.verify_workload(w)
    b = oracle.verify_workload(w, rule="always")
    np.testing.assert_array_equal(a.num_accepted, b.num_accepted)
    np.testing.assert_array_equal(a.next_token, b.next_token)


@pytest.mark.parametrize("alpha", [0.5, 2.0, 4.0])
def test_bild_discrepancy_is_the_cross_entropy(alpha):
    """BiLD*'s delta = 1(D(q, p) > alpha) with D = -sum_v q log p = H(q) + KL(q || p)
    (scipy.stats.entropy), the temperature-sampling discrepancy of the experiments."""
    from scipy.stats import entropy
    w = synthetic(12, 4, 500, dtype="f32", kind="gauss", sigma=1.0, rule="bild", alpha=alpha,
                  temperature=0.8, seed=61)
    r = oracle.verify_workload(w)
    decided = 0
    for b in range(w.B):
        for j in range(w.gamma):
            q = np_softmax(logits_as_f64(w.draft[b, j], "f32"), 0.8)
            p = np_softmax(logits_as_f64(w.target[b, j], "f32"), 0.8)
            D = entropy(q) + entropy(q, p)
            if abs(D - alpha) < 1e-9:
                continue
            assert r.row("delta")[b, j] == (1.0 if D > alpha else 0.0), (b, j, D)
            decided += 1
    assert decided == w.B * w.gamma
    # a threshold above every discrepancy defers nothing: every draft is accepted
    big = oracle.verify_workload(w, alpha=1e6)
    assert np.all(big.num_accepted == w.gamma)


# ----------------------------------------------------------------- log-loss rules, greedy decoding

@pytest.mark.parametrize("rule,alpha", [("chow_log", 2.0), ("chow_log", 3.5), ("diff_log", 0.2),
                                        ("opt_log", 0.5), ("opt_log", 2.0)])
def test_log_loss_rules_use_the_entropies(rule, alpha):
    """ChowLog: H(q) > alpha; DiffLog: -H(q) < -H(p) - alpha; OPTLog: -H(q) < -H(p) -
    alpha D_TV(p, q) (the log-loss plug-in rules), with H from scipy.stats.entropy."""
    from scipy.stats import entropy
    w = synthetic(10, 4, 300, dtype="f32", kind="gauss", sigma=1.0, rule=rule, alpha=alpha,
                  temperature=1.2, seed=71)
    r = oracle.verify_workload(w)
    for b in range(w.B):
        for j in range(w.gamma):
            q = np_softmax(logits_as_f64(w.draft[b, j], "f32"), 1.2)
            p = np_softmax(logits_as_f64(w.target[b, j], "f32"), 1.2)
            hq, hp, tv = entropy(q), entropy(p), 0.5 * np.abs(p - q).sum()
            lhs, rhs = {"chow_log": (hq, alpha), "diff_log": (-hq, -hp - alpha),
                        "opt_log": (-hq, -hp - alpha * tv)}[rule]
            want = lhs > rhs if rule == "chow_log" else lhs < rhs
            if abs(lhs - rhs) > 1e-9:
                assert r.row("delta")[b, j] == float(want), (b, j, lhs, rhs)


def _greedy_spec_decoding(w):
    """Greedy speculative decoding as its own procedure: a draft survives while it is
    the verifier's argmax; the first one that is not is replaced by the verifier's
    argmax, and after gamma survivors the bonus token is the argmax of p_gamma."""
    na, nt = [], []
    for b in range(w.B):
        p = logits_as_f64(w.target[b], w.dtype)
        for j in range(w.gamma + 1):
            ap = int(np.argmax(p[j]))
            if j == w.gamma or w.tokens[b, j] != ap:
                na.append(j)
                nt.append(ap)
                break
    return np.array(na), np.array(nt)


def test_greedy_always_defer_is_greedy_speculative_decoding():
    w = synthetic(16, 5, 400, dtype="bf16", kind="zipf", sigma=0.3, rule="always", alpha=0.0,
                  temperature=0.0, seed=81)
    r = oracle.verify_workload(w)
    na, nt = _greedy_spec_decoding(w)
    np.testing.assert_array_equal(r.num_accepted, na)
    np.testing.assert_array_equal(r.next_token, nt)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_greedy_bild_uses_the_log_probability_of_q_argmax(seed):
    """At T = 0 the BiLD baseline's discrepancy is D = -log p(argmax q) (lowest index
    on ties), not the sampling analogue -sum q log p: delta = [D > alpha] per row."""
    rng = np.random.default_rng(seed)
    g, V = 6, 50
    q_log = (rng.standard_normal((g, V)) * 2.0).astype(np.float32)
    p_log = (q_log[np.r_[0:g, g - 1]] + rng.standard_normal((g + 1, V)) * 1.5).astype(np.float32)
    q = np_softmax(q_log.astype(np.float64), 1.0)
    p = np_softmax(p_log.astype(np.float64), 1.0)
    D = -np.log(p[np.arange(g), q.argmax(1)])
    alpha = float(np.median(D))
    w = rows_workload(np.exp(q_log), np.exp(p_log), q_log.argmax(1), np.full(g + 1, 0.5), "bild", alpha)
    w.temperature = 0.0
    r = oracle.verify_workload(w)
    np.testing.assert_array_equal(r.row("delta")[0], (D > alpha).astype(float))
    assert 0 < (D > alpha).sum() < g


@pytest.mark.parametrize("alpha", [0.0, 0.05, 0.2, 0.6, 1.0])
def test_greedy_opt_equals_greedy_diff(alpha):
    """The greedy special case (appendix): with T -> 0 the OPT rule's TV term is
    1(argmax q != argmax p), and running OPT is equivalent to running Diff."""
    w = synthetic(32, 4, 300, dtype="f32", kind="gauss", sigma=1.0, rule="opt", alpha=alpha,
                  temperature=0.0, seed=91)
    a = oracle.verify_workload(w)
    d = oracle.verify_workload(w, rule="diff")
    np.testing.assert_array_equal(a.num_accepted, d.num_accepted)
    np.testing.assert_array_equal(a.next_token, d.next_token)
    assert np.all(a.status == 0)


def test_lossy_at_alpha_1_is_the_limit_of_alpha_below_1():
    """Table 3 / Lemma 2 at alpha = 1, read as the limit alpha -> 1-: the acceptance
    min(1, p(x)/((1 - alpha) q(x))) tends to 1 where p(x) > 0 and stays 0 where
    p(x) = 0 (a masked target logit), so the oracle at alpha = 1 decides as it does
    at alpha = 1 - 1e-12 and rejects exactly the drafts whose target logit is masked."""
    w = synthetic(12, 4, 300, dtype="f32", kind="gauss", sigma=1.0, rule="lossy", alpha=1.0, seed=81)
    for b in range(0, 12, 2):          # mask the target logit of one draft token per even sequence
        j = b % 4
        w.target[b, j, w.tokens[b, j]] = -np.inf
    one = oracle.verify_workload(w, alpha=1.0)
    near = oracle.verify_workload(w, alpha=1.0 - 1e-12)
    np.testing.assert_array_equal(one.num_accepted, near.num_accepted)
    np.testing.assert_array_equal(one.next_token, near.next_token)
    np.testing.assert_array_equal(one.row("accept"), near.row("accept"))
    for b in range(12):
        first_masked = b % 4 if b % 2 == 0 else w.gamma
        assert one.num_accepted[b] == first_masked, b


@pytest.mark.parametrize("gap", [50.0, 2000.0])
def test_bild_discrepancy_is_infinite_where_p_is_zero_and_q_is_not(gap):
    """D(q, p) = -sum_v q(v) log p(v) is +infinity as soon as one token has q(v) > 0
    and p(v) = 0: any finite draft logit gives q(v) > 0, a -inf target logit p(v) = 0.
    Here that token's draft logit lies `gap` below the row's largest, so q(v) is
    tiny (50) or below fp64's range (2000, exp(-2000) = 0): BiLD* defers
    (delta = 1) for any alpha either way, and does not where the masked target
    token's draft logit is masked too."""
    V, g = 5, 1
    q = np.array([[0.0, 1.0, -0.5, -gap, 0.3]], dtype=np.float32)
    p = np.array([[0.2, 0.9, -0.1, -np.inf, 0.0], [0.1, 0.2, 0.3, 0.4, 0.5]], dtype=np.float32)
    for alpha in (0.5, 50.0, 1e6):
        w = rows_workload(np.exp(q.astype(np.float64)), np.exp(p.astype(np.float64)), [1], [0.5, 0.5], "bild", alpha)
        w.draft[0] = q
        w.target[0] = p
        r = oracle.verify_workload(w)
        assert r.row("delta")[0, 0] == 1, (gap, alpha)
        w.draft[0, 0, 3] = -np.inf   # now q(3) = 0 too: D is finite, about 1.4 nats
        r = oracle.verify_workload(w)
        assert r.row("delta")[0, 0] == (1 if alpha < 1.0 else 0), (gap, alpha)


def test_lossy_rejection_with_an_empty_residual():
    """Lemma 2 with beta > 1: q = (1/2, 1/2), p = (0, 1), alpha = 0, beta = 2 give
    pi = max{min{q, p}, p/2} = (0, 1/2), so the draft x = 0 is rejected (pi/q = 0),
    while max(0, p/beta - q) = (0, 0) leaves no token to draw: next_token is -1,
    num_accepted 0, and the sequence is flagged (no draw to compare)."""
    w = rows_workload([[0.5, 0.5]], [[0.0, 1.0], [0.5, 0.5]], [0], [0.3, 0.7], "lossy", 0.0)
    r = oracle.verify_workload(w, beta=2.0)
    assert (r.num_accepted[0], r.next_token[0]) == (0, -1)
    assert r.flagged[0]
    # beta = 1: the residual is norm(max(0, p - q)) = (0, 1), token 1
    r1 = oracle.verify_workload(w, beta=1.0)
    assert (r1.num_accepted[0], r1.next_token[0]) == (0, 1) and not r1.flagged[0]
