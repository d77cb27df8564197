"""Pins of the float64 oracle to the paper and to independent mathematics.

Every check here compares the oracle with something other than itself: a
closed form, a library routine (scipy), a separately written textbook
algorithm, brute-force enumeration, or an exact sampling law tested by
chi-square.  No GPU is needed.
"""
import itertools
import math

import numpy as np
import pytest
from scipy.spatial.distance import jensenshannon
from scipy.special import log_softmax as sp_log_softmax
from scipy.special import softmax as sp_softmax
from scipy.stats import chisquare

import oracle as O


def rows_of(a, b, t, gamma=0.5, beta=1.0, div=O.DIV_JSD, lam=0.1, tokens=None,
            delta=O.DELTA_AB):
    K1 = a.shape[0]
    out = []
    for k in range(K1):
        d = int(tokens[k]) if tokens is not None and k < len(tokens) else None
        out.append(O.row_quantities(a[k], b[k], t[k], gamma, beta, div, lam, d, delta))
    return out


# ------------------------------------------------------------ log-softmax / LSE

def test_log_softmax_uniform_row_is_minus_log_v():
    for V in (2, 7, 32000):
        la = O.log_softmax(np.full(V, 3.25))
        assert np.allclose(la, -math.log(V), rtol=0, atol=1e-13)


def test_log_softmax_two_token_closed_form():
    for x in (-30.0, -1.5, 0.0, 0.7, 12.0):
        la = O.log_softmax(np.array([0.0, x]))
        z = math.log1p(math.exp(x)) if x < 30 else x
        assert la[0] == pytest.approx(-z, abs=1e-14)
        assert la[1] == pytest.approx(x - z, abs=1e-14)


def test_log_softmax_matches_scipy(rng):
    for V in (3, 1000, 151936):
        z = rng.normal(0, 4, V)
        assert np.allclose(O.log_softmax(z), sp_log_softmax(z), atol=1e-12, rtol=0)


# ------------------------------------------------------------ JSD (Eq. 3)

def test_jsd_closed_form_half_half_vs_point_mass():
    # p = (1/2, 1/2), q = (1, 0): m = (3/4, 1/4), KL(p||m) = 1/2 ln(4/3),
    # KL(q||m) = ln(4/3), JSD = 3/4 ln(4/3).
    la = np.log([0.5, 0.5])
    lb = np.array([0.0, -np.inf])
    with np.errstate(divide="ignore", invalid="ignore"):
        assert O.jsd(la, lb) == pytest.approx(0.75 * math.log(4 / 3), abs=1e-15)


def test_jsd_disjoint_supports_is_ln2():
    with np.errstate(divide="ignore", invalid="ignore"):
        assert O.jsd(np.array([0.0, -np.inf]), np.array([-np.inf, 0.0])) == pytest.approx(math.log(2), abs=1e-15)
    # finite logits approaching disjoint supports (the gate's lower bound gamma/2)
    a = np.array([[0.0, -1e4]])
    b = np.array([[-1e4, 0.0]])
    r = rows_of(a, b, a)[0]
    assert r.D == pytest.approx(math.log(2), abs=1e-12)
    assert r.gamma_eff == pytest.approx(0.25, abs=1e-12)


def test_jsd_two_point_entropy_form(rng):
    # JSD(P||Q) = H(M) - (H(P) + H(Q)) / 2 with binary entropies in nats.
    def H(x):
        return -sum(v * math.log(v) for v in (x, 1 - x) if v > 0)
    for _ in range(200):
        x, y = rng.uniform(0.001, 0.999, 2)
        want = H((x + y) / 2) - (H(x) + H(y)) / 2
        got = O.jsd(np.log([x, 1 - x]), np.log([y, 1 - y]))
        assert got == pytest.approx(want, abs=1e-14)


def test_jsd_matches_scipy_jensenshannon(rng):
    for V in (2, 8, 500, 32000):
        a = rng.normal(0, 2, V)
        b = a + rng.normal(0, 1.5, V)
        p, q = sp_softmax(a), sp_softmax(b)
        want = jensenshannon(p, q) ** 2          # natural log by default
        got = O.jsd(O.log_softmax(a), O.log_softmax(b))
        assert got == pytest.approx(want, rel=1e-9, abs=1e-14)


def test_jsd_symmetric_bounded_and_zero_iff_constant_shift(rng):
    for _ in range(50):
        V = int(rng.integers(2, 64))
        a = rng.normal(0, 3, V)
        b = rng.normal(0, 3, V)
        la, lb = O.log_softmax(a), O.log_softmax(b)
        d1, d2 = O.jsd(la, lb), O.jsd(lb, la)
        assert d1 == pytest.approx(d2, abs=1e-15)
        assert 0.0 < d1 <= math.log(2)
        # a - b constant  =>  identical distributions  =>  D = 0
        assert O.jsd(O.log_softmax(a), O.log_softmax(a + 5.5)) == pytest.approx(0.0, abs=1e-14)


# ------------------------------------------------------------ gate (Eq. 3, App. A)

def test_gate_range_monotone_and_zero_divergence(rng):
    B, K, V = 6, 3, 300
    gamma = 0.5
    a = rng.normal(0, 2, (B, K + 1, V))
    scale = np.linspace(0, 6, B)[:, None, None]
    b = a + scale * rng.normal(0, 1, (B, K + 1, V))
    t = rng.normal(0, 2, (B, K + 1, V))
    tokens = rng.integers(0, V, (B, K))
    res = O.fuse_verify(a.astype(np.float32), b.astype(np.float32), t.astype(np.float32),
                        tokens, gamma=gamma)
    D, g = res.D.ravel(), res.gamma_eff.ravel()
    assert np.all(g <= gamma + 1e-15) and np.all(g >= gamma / 2 - 1e-15)
    order = np.argsort(D)
    assert np.all(np.diff(g[order]) <= 1e-15)          # non-increasing in D
    # first batch element has identical contexts: zero divergence, zero gate
    assert np.allclose(res.D[0], 0.0, atol=1e-14)
    assert np.allclose(res.gamma_eff[0], gamma, atol=1e-14)
    # multiplicative composition (App. A) of the values the oracle produced:
    # gamma_eff(D1) * gamma_eff(D2) / gamma equals gamma * exp(-(D1 + D2)).
    for i, j in rng.integers(0, D.size, (20, 2)):
        assert g[i] * g[j] / gamma == pytest.approx(gamma * math.exp(-(D[i] + D[j])), rel=1e-14)


# ------------------------------------------------------------ fusion (Eq. 2)

def test_fused_target_probability_space_route(rng):
    # softmax(t + beta (a - b)) is proportional to softmax(t) (softmax(a) / softmax(b))^beta
    for beta in (0.0, 0.5, 1.0, 2.0):
        V = 64
        a, b, t = (rng.normal(0, 2, (1, V)) for _ in range(3))
        r = rows_of(a, b, t, beta=beta)[0]
        w = sp_softmax(t[0]) * (sp_softmax(a[0]) / sp_softmax(b[0])) ** beta
        assert np.allclose(np.exp(r.lq), w / w.sum(), atol=1e-15, rtol=1e-12)


def test_zero_delta_or_zero_beta_gives_verifier_distribution(rng):
    V = 1000
    a = rng.normal(0, 2, (1, V))
    t = rng.normal(0, 2, (1, V))
    r = rows_of(a, a.copy(), t, beta=1.0)[0]            # z_c == z_f
    assert np.allclose(r.lq, sp_log_softmax(t[0]), atol=1e-12, rtol=0)
    assert r.D == pytest.approx(0.0, abs=1e-14) and r.gamma_eff == pytest.approx(0.5, abs=1e-15)
    b = a + rng.normal(0, 3, (1, V))
    r = rows_of(a, b, t, beta=0.0)[0]
    assert np.allclose(r.lq, sp_log_softmax(t[0]), atol=1e-12, rtol=0)


def test_delta_sources_probability_space_routes(rng):
    # raw-augmented: softmax(t + beta a) is proportional to softmax(t) softmax(a)^beta;
    # SCD-style: softmax(t + beta (t - b)) to softmax(t)^(1 + beta) / softmax(b)^beta
    V = 64
    for beta in (0.0, 0.5, 1.0, 2.0):
        a, b, t = (rng.normal(0, 2, (1, V)) for _ in range(3))
        r = rows_of(a, b, t, beta=beta, delta=O.DELTA_A)[0]
        w = sp_softmax(t[0]) * sp_softmax(a[0]) ** beta
        assert np.allclose(np.exp(r.lq), w / w.sum(), atol=1e-15, rtol=1e-12)
        r = rows_of(a, b, t, beta=beta, delta=O.DELTA_TB)[0]
        w = sp_softmax(t[0]) ** (1.0 + beta) / sp_softmax(b[0]) ** beta
        assert np.allclose(np.exp(r.lq), w / w.sum(), atol=1e-15, rtol=1e-12)


def test_delta_sources_coincide_where_the_definitions_do(rng):
    B, K, V = 4, 3, 300
    a, b, t = (rng.normal(0, 2, (B, K + 1, V)).astype(np.float32) for _ in range(3))
    tokens = rng.integers(0, V, (B, K))
    # b constant along each row: a - b and a differ by a per-row constant
    flat = np.broadcast_to(b[..., :1], b.shape).copy()
    for mode in (O.GREEDY, O.STOCHASTIC):
        probs = np.full((B, K), 0.3, np.float32)
        unif = rng.random((B, K + 1)).astype(np.float32)
        kw = dict(mode=mode, want_logprobs=True, draft_probs=probs, uniforms=unif)
        r_ab = O.fuse_verify(a, flat, t, tokens, delta_source=O.DELTA_AB, **kw)
        r_a = O.fuse_verify(a, flat, t, tokens, delta_source=O.DELTA_A, **kw)
        assert np.allclose(r_ab.logprobs, r_a.logprobs, atol=1e-12, rtol=0)
        assert np.array_equal(r_ab.accept_len, r_a.accept_len)
        assert np.array_equal(r_ab.next_token, r_a.next_token)
        # a == t: a - b and t - b are the same signal
        r_ab = O.fuse_verify(t, b, t, tokens, delta_source=O.DELTA_AB, **kw)
        r_tb = O.fuse_verify(t, b, t, tokens, delta_source=O.DELTA_TB, **kw)
        assert np.array_equal(r_ab.logprobs, r_tb.logprobs)
        assert np.array_equal(r_ab.next_token, r_tb.next_token)


def test_delta_source_leaves_the_gate_and_greedy_acceptance_alone(rng):
    # Eq. 4 and Eq. 3 use a, b and t themselves: per-draft decisions, D and
    # gamma_eff are the same whatever delta fuses the emission; beta = 0
    # removes delta altogether
    B, K, V = 6, 3, 200
    a, b, t = (rng.normal(0, 2, (B, K + 1, V)).astype(np.float32) for _ in range(3))
    tokens = rng.integers(0, V, (B, K))
    base = O.fuse_verify(a, b, t, tokens)
    for src in (O.DELTA_A, O.DELTA_TB):
        r = O.fuse_verify(a, b, t, tokens, delta_source=src)
        assert np.array_equal(r.accept, base.accept)
        assert np.array_equal(r.D, base.D) and np.array_equal(r.gamma_eff, base.gamma_eff)
        assert np.array_equal(r.accept_len, base.accept_len)
        z = O.fuse_verify(a, b, t, tokens, delta_source=src, beta=0.0)
        z0 = O.fuse_verify(a, b, t, tokens, beta=0.0)
        assert np.array_equal(z.next_token, z0.next_token)
    with pytest.raises(ValueError):
        O.row_quantities(a[0, 0], b[0, 0], t[0, 0], 0.5, 1.0, O.DIV_JSD, delta_source=3)


def test_row_constant_shifts_change_nothing(rng):
    B, K, V = 3, 2, 200
    a, b, t = (rng.normal(0, 2, (B, K + 1, V)).astype(np.float32) for _ in range(3))
    tokens = rng.integers(0, V, (B, K))
    probs = rng.uniform(0.01, 1, (B, K)).astype(np.float32)
    unif = rng.uniform(0, 1, (B, K + 1)).astype(np.float32)
    shift = lambda x, c: (x + np.float32(c)).astype(np.float32)  # noqa: E731
    for mode in (O.GREEDY, O.STOCHASTIC):
        r0 = O.fuse_verify(a, b, t, tokens, probs, unif, mode=mode, want_logprobs=True)
        r1 = O.fuse_verify(shift(a, 4), shift(b, -2), shift(t, 8), tokens, probs, unif,
                           mode=mode, want_logprobs=True)
        assert np.allclose(r0.logprobs, r1.logprobs, atol=1e-5)
        assert np.allclose(r0.D, r1.D, atol=1e-6)
        ok = ~(r0.flagged | r1.flagged)
        assert np.array_equal(r0.accept_len[ok], r1.accept_len[ok])
        assert np.array_equal(r0.next_token[ok], r1.next_token[ok])


# ------------------------------------------------------------ Algorithm 1, brute force

def algorithm1_textbook(a, b, t, d, gamma, beta, fuse_bonus=False):
    """Algorithm 1 written out in probability space with scipy routines."""
    K = len(d)
    for i in range(K):
        p_a, p_b, p_t = sp_softmax(a[i]), sp_softmax(b[i]), sp_softmax(t[i])
        D = jensenshannon(p_a, p_b) ** 2
        g = gamma * math.exp(-D)
        if p_t[d[i]] > g * p_b[d[i]]:
            continue
        return i, int(np.argmax(t[i] + beta * (a[i] - b[i])))
    last = t[K] + beta * (a[K] - b[K]) if fuse_bonus else t[K]
    return K, int(np.argmax(last))


@pytest.mark.parametrize("V,K", [(2, 1), (3, 2), (5, 3), (8, 2), (8, 3)])
def test_greedy_brute_force_all_draft_tuples(rng, V, K):
    for trial in range(4):
        a = rng.normal(0, 1.5, (K + 1, V))
        b = a + rng.normal(0, 1.0 + trial, (K + 1, V))
        t = b + rng.normal(0, 1.0, (K + 1, V))
        gamma, beta = [(0.5, 1.0), (0.3, 0.5), (0.9, 2.0), (1.0, 0.0)][trial]
        fuse_bonus = bool(trial % 2)
        rows = rows_of(a, b, t, gamma=gamma, beta=beta)
        tuples = np.array(list(itertools.product(range(V), repeat=K)))
        L, nxt, flag, _, _ = O.greedy_scan(rows, tuples, K, fuse_bonus)
        for n, d in enumerate(tuples):
            if flag[n]:
                continue
            want = algorithm1_textbook(a, b, t, d, gamma, beta, fuse_bonus)
            assert (L[n], nxt[n]) == want, (trial, d)


def test_greedy_identical_verifier_and_compressed_drafter_accepts_all(rng):
    # t == b: softmax(t)[d] / softmax(b)[d] = 1 > gamma_eff whenever gamma_eff < 1
    B, K, V = 5, 4, 300
    a = rng.normal(0, 2, (B, K + 1, V)).astype(np.float32)
    b = (a + rng.normal(0, 2, (B, K + 1, V))).astype(np.float32)
    tokens = rng.integers(0, V, (B, K))
    res = O.fuse_verify(a, b, b.copy(), tokens, gamma=0.99)
    assert np.all(res.accept_len == K)
    assert np.array_equal(res.next_token, np.argmax(b[:, K], axis=1))


def test_beta0_gamma1_reading_of_the_degenerate_case(rng):
    # With beta = 0 and gamma = 1 the rule is p_t(d) > exp(-D) p_b(d) and the
    # emission at a rejection is the plain verifier argmax.
    K, V = 3, 50
    a, b, t = (rng.normal(0, 2, (K + 1, V)) for _ in range(3))
    rows = rows_of(a, b, t, gamma=1.0, beta=0.0)
    for d in rng.integers(0, V, (200, K)):
        L, nxt, flag, acc, _ = O.greedy_scan(rows, d[None, :], K)
        if flag[0]:
            continue
        for k in range(K):
            r = rows[k]
            stated = np.exp(r.lt[d[k]]) > math.exp(-r.D) * np.exp(r.lb[d[k]])
            assert acc[0, k] == stated
        if L[0] < K:
            assert nxt[0] == np.argmax(t[L[0]])


# ------------------------------------------------------------ stochastic extension

def textbook_speculative_sampling(p_rows, q_rows, d, u):
    """Leviathan et al. / Chen et al. speculative sampling, one step.

    p_rows: drafter distributions, q_rows: target distributions (K+1 rows),
    d: K drafts, u: K+1 uniforms (u[K] drives the one non-draft draw).
    """
    K = len(d)
    for i in range(K):
        p, q = p_rows[i], q_rows[i]
        if u[i] < min(1.0, q[d[i]] / p[d[i]]):
            continue
        r = np.maximum(q - p, 0.0)
        c = np.cumsum(r / r.sum())
        return i, int(min(np.searchsorted(c, u[K], side="right"), len(c) - 1))
    c = np.cumsum(q_rows[K])
    return K, int(min(np.searchsorted(c, u[K] * c[-1], side="right"), len(c) - 1))


def test_stochastic_zero_delta_gamma1_is_textbook_speculative_sampling(rng):
    K, V = 3, 40
    hits = 0
    for trial in range(30):
        a = rng.normal(0, 1.5, (K + 1, V))
        t = a + rng.normal(0, 1.0, (K + 1, V))
        rows = rows_of(a, a.copy(), t, gamma=1.0, beta=1.0)   # z_c == z_f: delta == 0
        p_rows = [sp_softmax(x) for x in a]
        q_rows = [sp_softmax(x) for x in t]
        N = 200
        d = np.stack([[rng.choice(V, p=p_rows[k]) for k in range(K)] for _ in range(N)])
        probs = np.array([[p_rows[k][d[n, k]] for k in range(K)] for n in range(N)])
        u = rng.uniform(0, 1, (N, K + 1))
        L, nxt, flag, _, _ = O.stochastic_scan(rows, d, probs, u, K)
        for n in range(N):
            if flag[n]:
                continue
            assert (L[n], nxt[n]) == textbook_speculative_sampling(p_rows, q_rows, d[n], u[n])
            hits += 1
    assert hits > 5000


def test_stochastic_identical_draft_and_target_accepts_everything(rng):
    # t + beta (a - b) == a + c  =>  fused target == drafter  =>  ratio == 1 > u gamma_eff
    B, K, V = 4, 5, 500
    beta = 1.0
    a = rng.normal(0, 2, (B, K + 1, V))
    b = a + rng.normal(0, 1, (B, K + 1, V))
    t = a - beta * (a - b) + 3.0
    tokens = np.zeros((B, K), np.int64)
    probs = np.zeros((B, K), np.float32)
    for bi in range(B):
        for k in range(K):
            p = sp_softmax(a[bi, k])
            tokens[bi, k] = rng.choice(V, p=p)
            probs[bi, k] = p[tokens[bi, k]]
    unif = rng.uniform(0, 1, (B, K + 1)).astype(np.float32)
    unif[:, :K] = np.float32(0.999999)
    res = O.fuse_verify(a, b, t, tokens, probs, unif, mode=O.STOCHASTIC, gamma=1.0, beta=beta)
    ok = ~res.flagged
    assert ok.sum() >= B - 1
    assert np.all(res.accept_len[ok] == K)


def exact_first_token_law(rows, gamma_eff):
    """P(first emitted token = x) for K >= 1 (position 1 only).

    P(x) = p(x) A(x) + (1 - sum_y p(y) A(y)) r(x) / R with
    A(y) = min(1, q(y) / (gamma_eff p(y))), r = max(0, q - p).
    """
    r0 = rows[0]
    p = np.exp(r0.la)
    q = np.exp(r0.lq)
    A = np.minimum(1.0, q / (gamma_eff * p))
    resid = np.maximum(q - p, 0.0)
    return p * A + (1.0 - np.sum(p * A)) * resid / resid.sum()


@pytest.mark.parametrize("div,gamma", [(O.DIV_NONE, 1.0), (O.DIV_JSD, 0.5), (O.DIV_JSD, 1.0)])
def test_stochastic_first_token_law_chi_square(rng, div, gamma):
    V, K, N = 6, 1, 1_000_000
    a = rng.normal(0, 1.0, (K + 1, V))
    b = a + rng.normal(0, 1.0, (K + 1, V))
    t = rng.normal(0, 1.0, (K + 1, V))
    rows = rows_of(a, b, t, gamma=gamma, beta=1.0, div=div)
    p = np.exp(rows[0].la)
    d = np.minimum(np.searchsorted(np.cumsum(p), rng.uniform(0, 1, N), side="right"), V - 1)
    probs = p[d]
    u = rng.uniform(0, 1, (N, K + 1))
    L, nxt, _, _, _ = O.stochastic_scan(rows, d[:, None], probs[:, None], u, K)
    first = np.where(L >= 1, d, nxt)
    counts = np.bincount(first, minlength=V)
    law = exact_first_token_law(rows, rows[0].gamma_eff)
    assert chisquare(counts, law * N).pvalue > 1e-3
    if div == O.DIV_NONE and gamma == 1.0:
        # lossless: the emitted token follows the fused target exactly
        assert np.allclose(law, np.exp(rows[0].lq), atol=1e-14)
        assert chisquare(counts, np.exp(rows[0].lq) * N).pvalue > 1e-3


# ------------------------------------------------------------ gate variants

def test_kl_and_lambda_gates(rng):
    V = 400
    a = rng.normal(0, 2, (2, V))
    b = a + rng.normal(0, 2, (2, V))
    t = rng.normal(0, 2, (2, V))
    p, q = sp_softmax(a[0]), sp_softmax(b[0])
    r = rows_of(a, b, t, div=O.DIV_KL)[0]
    assert r.D == pytest.approx(float(np.sum(p * np.log(p / q))), rel=1e-12)
    d = 17
    r = rows_of(a, b, t, div=O.DIV_LAMBDA, lam=0.1, tokens=[d])[0]
    assert r.gamma_eff == pytest.approx(0.5 * math.exp(-0.1 * math.log(p[d] / q[d])), rel=1e-6)
    r = rows_of(a, b, t, div=O.DIV_NONE)[0]
    assert r.gamma_eff == 0.5


# ------------------------------------------------------------ data errors

def test_data_errors_are_reported_not_raised(rng):
    B, K, V = 4, 2, 30
    a, b, t = (rng.normal(0, 1, (B, K + 1, V)).astype(np.float32) for _ in range(3))
    a[1, 0, 3] = np.nan
    t[2, 2, 0] = np.inf
    tokens = rng.integers(0, V, (B, K))
    tokens[3, 1] = V
    res = O.fuse_verify(a, b, t, tokens)
    assert list(res.error) == [False, True, True, True]
    assert list(res.accept_len[1:]) == [-1, -1, -1] and list(res.next_token[1:]) == [-1, -1, -1]
    probs = np.full((B, K), 0.5, np.float32)
    unif = np.full((B, K + 1), 0.5, np.float32)
    a[1, 0, 3] = 0
    t[2, 2, 0] = 0
    tokens[3, 1] = 0
    probs[0, 0] = 0.0
    unif[1, 2] = 1.0
    res = O.fuse_verify(a, b, t, tokens, probs, unif, mode=O.STOCHASTIC)
    assert list(res.error) == [True, True, False, False]


# ------------------------------------------------------------ the drafter's draw

def test_draft_sample_greedy_ties_and_probability():
    # argmax with the lowest index among ties, and the closed-form probability
    a = np.array([[0.0, 2.0, 2.0, 1.0], [5.0, 5.0, 5.0, 5.0], [-1.0, -3.0, -2.0, -1.0]])
    r = O.draft_sample(a, mode=O.GREEDY)
    assert list(r.tokens) == [1, 0, 0]
    z = np.exp(2.0) * 2 + 1.0 + np.exp(1.0)
    assert r.probs[0] == pytest.approx(np.exp(2.0) / z, rel=1e-15)
    assert r.probs[1] == pytest.approx(0.25, rel=1e-15)
    assert list(r.flagged) == [True, True, True]   # every row here is an exact tie


def test_draft_sample_inverse_cdf_boundaries():
    # softmax = (0.1, 0.2, 0.3, 0.4): cumulative 0.1, 0.3, 0.6, 1.0; the draw is
    # the smallest index whose cumulative mass exceeds u
    a = np.log(np.array([[0.1, 0.2, 0.3, 0.4]] * 6))
    u = np.array([0.0, 0.05, 0.1 + 1e-3, 0.299, 0.6 + 1e-3, 0.999], np.float32)
    r = O.draft_sample(a, u, mode=O.STOCHASTIC)
    assert list(r.tokens) == [0, 0, 1, 1, 3, 3]
    # (the logits are stored as float32, so the probabilities are exact to ~1e-7)
    assert np.allclose(r.probs, [0.1, 0.1, 0.2, 0.2, 0.4, 0.4], rtol=1e-6, atol=0)
    assert not r.flagged[[1, 3, 5]].any() and r.flagged[0]   # u = 0 sits on the boundary 0


def test_draft_sample_law_chi_square(rng):
    V, N = 8, 1_000_000
    a = rng.normal(0, 1, (1, V))
    p = sp_softmax(a[0])
    u = rng.random(N).astype(np.float32)
    # the oracle's rule on one row, vectorised through inverse_cdf's targets
    idx, _ = O.inverse_cdf(np.exp(O.log_softmax(a[0])), u.astype(np.float64))
    counts = np.bincount(idx, minlength=V)
    assert chisquare(counts, N * p).pvalue > 1e-3
    r = O.draft_sample(np.repeat(a, 100, axis=0), u[:100], mode=O.STOCHASTIC)
    assert np.array_equal(r.tokens, idx[:100])


def test_draft_sample_shift_invariance_and_errors(rng):
    a = rng.normal(0, 2, (5, 300))
    u = rng.random(5).astype(np.float32)
    for mode in (O.GREEDY, O.STOCHASTIC):
        r0 = O.draft_sample(a, u, mode=mode)
        r1 = O.draft_sample(a + 7.25, u, mode=mode)
        assert np.array_equal(r0.tokens, r1.tokens)
        # the shifted logits are stored as float32 again: equal to its rounding
        assert np.allclose(r0.probs, r1.probs, rtol=1e-5, atol=0)
    bad = a.copy()
    bad[2, 7] = np.nan
    r = O.draft_sample(bad, u, mode=O.GREEDY)
    assert list(r.error) == [False, False, True, False, False] and r.tokens[2] == -1
    ub = u.copy()
    ub[4] = 1.0
    r = O.draft_sample(a, ub, mode=O.STOCHASTIC)
    assert r.error[4] and not r.error[:4].any()


# ------------------------------------------------- cross-family vocabularies

def _xcase(rng, B, K, V_d, V_v, S, scale=2.0):
    a = rng.normal(0, scale, (B, K + 1, V_d)).astype(np.float32)
    b = (a + rng.normal(0, 1.0, a.shape)).astype(np.float32)
    t = rng.normal(0, scale, (B, K + 1, V_v)).astype(np.float32)
    md = rng.choice(V_d, S, replace=False)
    mv = rng.choice(V_v, S, replace=False)
    draft = rng.integers(0, S, (B, K))
    probs = rng.uniform(0.05, 1.0, (B, K)).astype(np.float32)
    unif = rng.random((B, K + 1)).astype(np.float32)
    return a, b, t, md, mv, draft, probs, unif


def _same(r0, r1, next_map=None):
    assert np.array_equal(r0.accept_len, r1.accept_len)
    nt = r0.next_token if next_map is None else np.where(r0.next_token >= 0,
                                                          next_map[np.maximum(r0.next_token, 0)], -1)
    assert np.array_equal(nt, r1.next_token)
    assert np.array_equal(r0.flagged, r1.flagged) and np.array_equal(r0.error, r1.error)
    np.testing.assert_allclose(r0.D, r1.D, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("mode", [O.GREEDY, O.STOCHASTIC])
def test_xvocab_identity_map_is_the_plain_step(rng, mode):
    # one shared vocabulary, every token paired with itself
    a, b, t, _, _, draft, probs, unif = _xcase(rng, 3, 3, 40, 40, 40)
    ident = np.arange(40)
    r0 = O.fuse_verify(a, b, t, draft, probs, unif, mode=mode)
    r1 = O.fuse_verify_xvocab(a, b, t, ident, ident, draft, probs, unif, mode=mode)
    _same(r0, r1)
    assert np.array_equal(r1.next_index, r0.next_token)
    np.testing.assert_allclose(r0.lse, r1.lse, rtol=1e-12)


@pytest.mark.parametrize("mode", [O.GREEDY, O.STOCHASTIC])
def test_xvocab_tokens_outside_the_shared_set_do_not_matter(rng, mode):
    # committed tokens are restricted to the pairs: changing (even poisoning)
    # unpaired logits of either vocabulary changes nothing
    a, b, t, md, mv, draft, probs, unif = _xcase(rng, 4, 2, 70, 55, 30)
    r0 = O.fuse_verify_xvocab(a, b, t, md, mv, draft, probs, unif, mode=mode)
    free_d = np.setdiff1d(np.arange(70), md)
    free_v = np.setdiff1d(np.arange(55), mv)
    a2, b2, t2 = a.copy(), b.copy(), t.copy()
    a2[..., free_d] = 60.0
    b2[..., free_d] = np.nan
    t2[..., free_v] = rng.normal(30, 5, t2[..., free_v].shape)
    r1 = O.fuse_verify_xvocab(a2, b2, t2, md, mv, draft, probs, unif, mode=mode)
    _same(r0, r1)
    assert not r1.error.any()


@pytest.mark.parametrize("mode", [O.GREEDY, O.STOCHASTIC])
def test_xvocab_relabelling_either_vocabulary(rng, mode):
    # renaming the verifier's tokens renames the committed token and nothing
    # else; renaming the drafter's tokens changes nothing
    a, b, t, md, mv, draft, probs, unif = _xcase(rng, 4, 3, 64, 48, 36)
    r0 = O.fuse_verify_xvocab(a, b, t, md, mv, draft, probs, unif, mode=mode)
    pv = rng.permutation(48)
    t2 = np.empty_like(t)
    t2[..., pv] = t
    r1 = O.fuse_verify_xvocab(a, b, t2, md, pv[mv], draft, probs, unif, mode=mode)
    _same(r0, r1, next_map=pv)
    pd = rng.permutation(64)
    a2, b2 = np.empty_like(a), np.empty_like(b)
    a2[..., pd] = a
    b2[..., pd] = b
    r2 = O.fuse_verify_xvocab(a2, b2, t, pd[md], mv, draft, probs, unif, mode=mode)
    _same(r0, r2)


def test_xvocab_restricted_normalisation_closed_form():
    # two pairs, K = 1, greedy.  Over the pairs: p_a' = (1/2, 1/2),
    # p_b' = (0.8, 0.2), p_t' = (e^2, 1) / (e^2 + 1).  The unpaired verifier
    # tokens 0 and 3 carry almost all of the full verifier vocabulary's mass:
    # normalised over the full vocabulary the draft would be rejected
    # (p_t = 1 / (2 e^35 + e^2 + 1) against gamma_eff p_b ~ 0.1); over the pairs
    # it is accepted (1 / (1 + e^2) = 0.119 > gamma_eff 0.2).
    V_d, V_v = 3, 4
    md, mv = np.array([1, 0]), np.array([2, 1])
    a = np.zeros((1, 2, V_d), np.float32)
    a[..., 2] = -30.0
    b = np.zeros((1, 2, V_d), np.float32)
    b[..., 1], b[..., 0], b[..., 2] = np.log(0.8), np.log(0.2), -30.0
    t = np.zeros((1, 2, V_v), np.float32)
    t[..., 0] = t[..., 3] = 35.0
    t[0, :, 2], t[0, :, 1] = 2.0, 0.0          # t' = (2, 0)
    draft = np.array([[1]])                     # pair 1: drafter token 0, verifier token 1
    r = O.fuse_verify_xvocab(a, b, t, md, mv, draft, gamma=0.5, beta=1.0)
    p = np.array([0.5, 0.5])
    q = np.array([np.float32(np.log(0.8)), np.float32(np.log(0.2))], np.float64)
    q = np.exp(q) / np.exp(q).sum()
    m = (p + q) / 2
    D = 0.5 * np.sum(p * np.log(p / m)) + 0.5 * np.sum(q * np.log(q / m))
    assert r.D[0, 0] == pytest.approx(D, rel=1e-9)
    gamma_eff = 0.5 * np.exp(-D)
    assert r.gamma_eff[0, 0] == pytest.approx(gamma_eff, rel=1e-7)
    pt = 1.0 / (1.0 + np.exp(2.0))
    assert pt > gamma_eff * q[1] and r.accept_len[0] == 1
    assert 1.0 / (2 * np.exp(35.0) + np.exp(2.0) + 1.0) < gamma_eff * q[1]
    # all K drafts accepted: the bonus row emits argmax t' = pair 0 = verifier token 2
    assert r.next_index[0] == 0 and r.next_token[0] == 2


def test_xvocab_maps_and_draft_indices_are_validated(rng):
    a, b, t, md, mv, draft, probs, unif = _xcase(rng, 2, 2, 30, 20, 10)
    with pytest.raises(ValueError):
        O.fuse_verify_xvocab(a, b, t, md, mv[:-1], draft)
    bad = md.copy()
    bad[3] = bad[4]
    with pytest.raises(ValueError):
        O.fuse_verify_xvocab(a, b, t, bad, mv, draft)
    bad = mv.copy()
    bad[0] = 20
    with pytest.raises(ValueError):
        O.fuse_verify_xvocab(a, b, t, md, bad, draft)
    d2 = draft.copy()
    d2[1, 0] = 10                                # a pair index outside [0, S)
    r = O.fuse_verify_xvocab(a, b, t, md, mv, d2)
    assert list(r.error) == [False, True] and r.next_token[1] == -1
