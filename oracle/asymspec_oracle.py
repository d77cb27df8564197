"""Plain float64 CPU oracle of AsymSpec's per-step fuse-and-verify.

TEST INFRASTRUCTURE ONLY.  Nothing in the library imports this module; only
``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` leg of
``bench.py`` may use it.  It shares no code with the CUDA path.

What it computes, for each batch element and each of its K+1 rows (row k is
the paper's position i = k+1; row K is the position after the last draft):

* Eq. 1 (Section 3.2): the context-gain signal delta_i = a_i - b_i, where a is
  the drafter on the full context and b the drafter on the compressed one.
* Eq. 2: the delta-fused emission argmax(t_i + beta * delta_i), t being the
  verifier on the compressed context.  The fused distribution
  softmax(t_i + beta * delta_i) is reported as log-probabilities; it equals
  softmax(t + beta (log softmax a - log softmax b)) because the two forms of
  delta differ by a per-row constant.
* Eq. 3 (Section 3.3): D_i = JSD(softmax(a_i) || softmax(b_i)) in nats, and the
  effective threshold gamma_eff(i) = gamma * exp(-D_i), which lies in
  [gamma/2, gamma] because the JSD is at most ln 2 (Appendix A).
* Eq. 4 and Algorithm 1: greedy verification.  d_i is accepted iff
  softmax(t_i)[d_i] > gamma_eff(i) * softmax(b_i)[d_i]; at the first rejection
  the fused argmax of that position is emitted; if all K drafts pass, the
  verifier's argmax at position K+1 is emitted (or, with fuse_bonus, the fused
  argmax there).
* Stochastic extension (not in the paper, which decodes greedily; defined
  here as the standard speculative-sampling rule of Leviathan et al. and Chen
  et al., with the paper's CDA relaxation multiplying the uniform threshold):
  d_i is accepted iff q_i(d_i) / p_draft(d_i) > u_i * gamma_eff(i), where q_i
  is the fused distribution and p_draft the probability the drafter gave
  d_i.  At the first rejection the token is drawn from the residual
  max(0, q_i - softmax(a_i)) normalised (from q_i itself if that residual is
  identically zero) by inverse CDF at u_K; if all K drafts pass, the token
  is drawn from q_{K+1} at u_K.
* Gate variants the paper compares in its ablations: no divergence (fixed
  gamma, Appendix B "fixed-gamma gate"), KL(softmax a || softmax b) in place of
  the JSD (Table "JSD vs KL"), and the tuned-lambda gate
  gamma * exp(-lambda * Delta) with Delta = log softmax(a_i)[d_i] -
  log softmax(b_i)[d_i] evaluated at the draft token (Appendix B).
* delta sources the paper's mechanism ablation (Section 5, "Mechanism
  ablation" table) compares with its own a - b: raw-augmented, delta = a (the
  drafter's full-context logits alone), and SCD-style, delta = t - b (the
  verifier against the compressed drafter).  Only the fused scores change;
  the gate and the acceptance test of Eq. 4 keep their own a, b and t.

* Cross-family vocabularies (Section 4, "Cross-family portability", and the
  appendix of the same name): drafter and verifier with different
  vocabularies share S string-identical tokens, the pairs (map_d[j],
  map_v[j]).  delta is computed in the drafter vocabulary and carried to the
  verifier token of each pair, and committed tokens are restricted to the
  shared set.  Read here as: the step above run on the rows restricted to
  the pairs, a'_j = a[map_d[j]], b'_j = b[map_d[j]], t'_j = t[map_v[j]]
  (every softmax, the divergence, the acceptance test and the emission
  renormalised over the shared set, index order = pair order), drafts given
  as pair indices, and the emitted pair index reported as its verifier token.

Near-ties.  Every decision the step takes from floating-point values (an
acceptance test, an argmax, an inverse-CDF boundary) is also measured here in
float64; a decision closer to its boundary than the bands below is "flagged"
and a batch element whose reached decisions include a flagged one is reported
as such, so that a float32 implementation may legitimately differ there:

* acceptance: |u - ratio / gamma_eff| < 1e-6, with u = 1 in greedy mode and
  ratio = softmax(t)[d] / softmax(b)[d] (greedy) or q(d) / p_draft (stochastic);
* argmax: gap between the two largest scores < 1e-6 * max(1, |largest|);
* inverse CDF: the target u * mass within CDF_BAND = 5e-7 (in units of
  probability mass) of either neighbouring cumulative boundary, or the
  residual mass itself below CDF_BAND.  An fp32 implementation's cumulative
  position error is dominated by the float32 rounding of the two
  normalisers the residual max(0, q - p) is built from: each (in log2 units,
  of magnitude below 32) carries at most 2^-20 of rounding, a relative mass
  error of at most 2^-20 ln 2 = 6.6e-7, and the position error is their
  difference times the part of the fused mass between the boundary and the
  target, a fraction of the total; the blocked float32 prefix adds about
  2^-24 per level of the summation tree.

Inputs are required to be finite (the paper's setting); a batch element with a
non-finite logit in the data the step uses, a draft token outside [0, V), or
(stochastic mode) a draft probability outside (0, 1] or a uniform outside
[0, 1) is reported as a data error with accept_len = next_token = -1.  Greedy
decoding without a fused bonus does not use a and b of the bonus row.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

GREEDY = 0
STOCHASTIC = 1

DIV_JSD = 0
DIV_NONE = 1
DIV_KL = 2
DIV_LAMBDA = 3

DELTA_AB = 0   # delta = a - b (Eq. 1, the paper's)
DELTA_A = 1    # delta = a (raw-augmented, mechanism ablation)
DELTA_TB = 2   # delta = t - b (SCD-style, mechanism ablation)

FP32 = 0
BF16 = 1

ACCEPT_BAND = 1e-6
ARGMAX_BAND = 1e-6
CDF_BAND = 5e-7
LN2 = float(np.log(2.0))


def widen(x: np.ndarray, dtype: int) -> np.ndarray:
    """Exact conversion of the stored logits to float64 (bf16 = uint16 bits)."""
    if dtype == BF16:
        bits = np.asarray(x, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
        return bits.view(np.float32).astype(np.float64)
    return np.asarray(x, dtype=np.float32).astype(np.float64)


# ----------------------------------------------------------- row quantities

def log_softmax(z: np.ndarray) -> np.ndarray:
    """log softmax(z) with the max shift, in float64."""
    m = np.max(z)
    return z - (m + np.log(np.sum(np.exp(z - m))))


def logsumexp(z: np.ndarray) -> float:
    m = np.max(z)
    return float(m + np.log(np.sum(np.exp(z - m))))


def jsd(la: np.ndarray, lb: np.ndarray) -> float:
    """Eq. 3: JSD(P || Q) in nats from the log-probabilities of P and Q.

    JSD = 1/2 KL(P || M) + 1/2 KL(Q || M), M = (P + Q) / 2, summed
    token by token as 1/2 [p (log p - log m) + q (log q - log m)], where a
    token with zero mass in P (or Q) contributes nothing for that term.
    """
    p = np.exp(la)
    q = np.exp(lb)
    with np.errstate(invalid="ignore"):
        lm = np.logaddexp(la, lb) - LN2
    tp = np.where(p > 0.0, p * (la - lm), 0.0)
    tq = np.where(q > 0.0, q * (lb - lm), 0.0)
    return float(0.5 * np.sum(tp + tq))


def kl(la: np.ndarray, lb: np.ndarray) -> float:
    """KL(P || Q) in nats, zero-mass tokens of P contributing nothing."""
    p = np.exp(la)
    return float(np.sum(np.where(p > 0.0, p * (la - lb), 0.0)))


def argmax_first(z: np.ndarray) -> int:
    """Index of the largest value, the lowest index among ties."""
    return int(np.argmax(z))


def top2_gap(z: np.ndarray) -> float:
    if z.size < 2:
        return np.inf
    top2 = np.partition(z, z.size - 2)[-2:]
    return float(top2[1] - top2[0])


def inverse_cdf(mass: np.ndarray, targets):
    """Smallest index y with sum_{z <= y} mass[z] > target, for each target.

    The cumulative sum runs in index order.  Returns (indices, distances),
    the distance being from the target to the nearer of the two cumulative
    boundaries around it.  If rounding leaves no such index, the last index
    with positive mass is returned with distance 0.
    """
    targets = np.atleast_1d(np.asarray(targets, np.float64))
    cum = np.cumsum(mass)
    y = np.searchsorted(cum, targets, side="right")
    over = y >= mass.size
    pos = np.nonzero(mass > 0.0)[0]
    last = int(pos[-1]) if pos.size else mass.size - 1
    yc = np.where(over, last, y)
    hi = cum[np.minimum(y, mass.size - 1)]
    lo = np.where(yc > 0, cum[np.maximum(yc - 1, 0)], 0.0)
    dist = np.where(over, 0.0, np.minimum(hi - targets, targets - lo))
    return yc.astype(np.int64), dist


@dataclass
class Row:
    """All per-row quantities of Eqs. 1-4 for one (b, k) position."""

    t: np.ndarray           # verifier logits
    la: np.ndarray          # log softmax(a)
    lb: np.ndarray          # log softmax(b)
    lt: np.ndarray          # log softmax(t)
    s: np.ndarray           # fused scores t + beta * delta (Eq. 2)
    lq: np.ndarray          # log softmax(s): the fused target
    lse_a: float
    lse_b: float
    lse_t: float
    lse_s: float
    D: float                # divergence of the selected gate
    gamma_eff: float


def row_quantities(a, b, t, gamma, beta, divergence, lam=0.1, draft_token=None,
                   delta_source=DELTA_AB) -> Row:
    """Eqs. 1-3 for one position (a, b, t are float64 logit rows)."""
    if delta_source == DELTA_AB:
        delta = a - b                               # Eq. 1
    elif delta_source == DELTA_A:
        delta = a                                   # raw-augmented (ablation)
    elif delta_source == DELTA_TB:
        delta = t - b                               # SCD-style (ablation)
    else:
        raise ValueError(f"unknown delta source {delta_source}")
    s = t + beta * delta                            # Eq. 2 (argument of argmax)
    lse_a, lse_b, lse_t, lse_s = logsumexp(a), logsumexp(b), logsumexp(t), logsumexp(s)
    la, lb, lt, lq = a - lse_a, b - lse_b, t - lse_t, s - lse_s
    if divergence == DIV_JSD:                       # Eq. 3, JSD in [0, ln 2]
        D = min(max(jsd(la, lb), 0.0), LN2)
    elif divergence == DIV_NONE:                    # fixed-gamma gate
        D = 0.0
    elif divergence == DIV_KL:                      # KL in place of the JSD
        D = max(kl(la, lb), 0.0)
    elif divergence == DIV_LAMBDA:                  # tuned-lambda gate
        D = lam * float(la[draft_token] - lb[draft_token]) if draft_token is not None else 0.0
    else:
        raise ValueError(f"unknown divergence {divergence}")
    gamma_eff = gamma * float(np.exp(-D))           # Eq. 3
    return Row(t, la, lb, lt, s, lq, lse_a, lse_b, lse_t, lse_s, D, gamma_eff)


# ----------------------------------------------------------- the scans

def greedy_candidates(rows, K: int, fuse_bonus: bool):
    """Token emitted if the scan stops at each row, and its near-tie flag.

    Rows k < K: the fused argmax (Eq. 2).  Row K: the verifier's argmax
    (Algorithm 1, the emission after all drafts pass), or the fused argmax
    with fuse_bonus.
    """
    cand = np.zeros(K + 1, np.int64)
    flag = np.zeros(K + 1, bool)
    for k, r in enumerate(rows):
        z = r.s if (k < K or fuse_bonus) else r.t
        cand[k] = argmax_first(z)
        flag[k] = top2_gap(z) < ARGMAX_BAND * max(1.0, abs(float(np.max(z))))
    return cand, flag


def greedy_scan(rows, tokens, K: int, fuse_bonus: bool = False):
    """Algorithm 1's verification loop for N draft tuples sharing the rows.

    tokens: [N, K].  Returns accept_len [N], next_token [N], flagged [N],
    accept [N, K] and margin [N, K] (margin = 1 - ratio / gamma_eff).
    """
    tokens = np.atleast_2d(np.asarray(tokens, np.int64))
    N = tokens.shape[0]
    cand, cflag = greedy_candidates(rows, K, fuse_bonus)
    accept = np.zeros((N, K), bool)
    margin = np.zeros((N, K))
    for k in range(K):
        r = rows[k]
        d = tokens[:, k]
        pt = np.exp(r.lt[d])                        # softmax(t_i)[d_i]
        pb = np.exp(r.lb[d])                        # softmax(b_i)[d_i]
        accept[:, k] = pt > r.gamma_eff * pb        # Eq. 4, strict
        margin[:, k] = 1.0 - np.exp(r.lt[d] - r.lb[d]) / r.gamma_eff
    return _finish_scan(accept, margin, cand, cflag, K)


def stochastic_candidates(rows, K: int, u_last):
    """Inverse-CDF draw at each row for N sampling uniforms u_K.

    Rows k < K draw from the residual max(0, q - softmax(a)) (from q if the
    residual is identically zero); row K draws from q.  Returns [N, K+1]
    tokens and near-tie flags.
    """
    u_last = np.atleast_1d(np.asarray(u_last, np.float64))
    N = u_last.size
    cand = np.zeros((N, K + 1), np.int64)
    flag = np.zeros((N, K + 1), bool)
    for k, r in enumerate(rows):
        q = np.exp(r.lq)
        if k < K:
            resid = np.maximum(q - np.exp(r.la), 0.0)
            R = float(np.sum(resid))
            mass = resid if R > 0.0 else q
            y, dist = inverse_cdf(mass, u_last * float(np.sum(mass)))
            cand[:, k] = y
            flag[:, k] = (dist < CDF_BAND) | (R < CDF_BAND)
        else:
            y, dist = inverse_cdf(q, u_last * float(np.sum(q)))
            cand[:, k] = y
            flag[:, k] = dist < CDF_BAND
    return cand, flag


def stochastic_scan(rows, tokens, probs, unif, K: int):
    """Speculative sampling with the CDA-relaxed threshold for N draws.

    tokens, probs: [N, K]; unif: [N, K+1] (unif[:, k] for the k-th test,
    unif[:, K] for the one inverse-CDF draw).  Returns as greedy_scan, with
    margin = u - ratio / gamma_eff.
    """
    tokens = np.atleast_2d(np.asarray(tokens, np.int64))
    probs = np.atleast_2d(np.asarray(probs, np.float64))
    unif = np.atleast_2d(np.asarray(unif, np.float64))
    N = tokens.shape[0]
    cand, cflag = stochastic_candidates(rows, K, unif[:, K])
    accept = np.zeros((N, K), bool)
    margin = np.zeros((N, K))
    for k in range(K):
        r = rows[k]
        ratio = np.exp(r.lq[tokens[:, k]]) / probs[:, k]
        accept[:, k] = ratio > unif[:, k] * r.gamma_eff      # strict
        margin[:, k] = unif[:, k] - ratio / r.gamma_eff
    return _finish_scan(accept, margin, cand, cflag, K)


def _finish_scan(accept, margin, cand, cflag, K):
    """First rejection stops the scan; flags count only reached decisions."""
    N = accept.shape[0]
    cand = np.broadcast_to(cand, (N, K + 1))
    cflag = np.broadcast_to(cflag, (N, K + 1))
    rejected = ~accept
    first = np.where(rejected.any(axis=1), rejected.argmax(axis=1), K)
    idx = np.arange(N)
    next_token = cand[idx, first]
    near = np.abs(margin) < ACCEPT_BAND
    reached = np.arange(K)[None, :] <= first[:, None]
    flagged = (near & reached).any(axis=1) | cflag[idx, first]
    return first.astype(np.int64), next_token.astype(np.int64), flagged, accept, margin


# ----------------------------------------------------------- the batch

@dataclass
class Result:
    accept_len: np.ndarray      # [B] int, -1 on data error
    next_token: np.ndarray      # [B] int, -1 on data error
    flagged: np.ndarray         # [B] bool: a reached decision is a near-tie
    error: np.ndarray           # [B] bool: data error
    lse: np.ndarray             # [B, K+1, 4] (a, b, t, s)
    D: np.ndarray               # [B, K+1]
    gamma_eff: np.ndarray       # [B, K+1]
    fused_argmax: np.ndarray    # [B, K+1] argmax of t + beta * delta
    fused_gap_flag: np.ndarray  # [B, K+1] that argmax is a near-tie
    candidate: np.ndarray       # [B, K+1] token emitted if the scan stops at this row
    cand_flag: np.ndarray       # [B, K+1] the candidate's own decision is a near-tie
    accept: np.ndarray          # [B, K] per-draft decisions
    accept_margin: np.ndarray   # [B, K]
    logprobs: np.ndarray | None  # [B, K+1, V] fused log-probs if requested


def fuse_verify(logits_full, logits_comp, logits_ver, draft_tokens, draft_probs=None,
                uniforms=None, *, dtype=FP32, gamma=0.5, beta=1.0, mode=GREEDY,
                divergence=DIV_JSD, lam=0.1, fuse_bonus=False,
                want_logprobs=False, delta_source=DELTA_AB) -> Result:
    """Runs the step over a batch.

    logits_*: [B, K+1, V] in the stored dtype (float32, or uint16 bf16 bits);
    draft_tokens: [B, K] int; draft_probs: [B, K] float32 and uniforms:
    [B, K+1] float32 (stochastic mode only).  gamma, beta and lambda are
    taken at float32 precision, the precision they are passed in.
    """
    gamma = float(np.float32(gamma))
    beta = float(np.float32(beta))
    lam = float(np.float32(lam))
    if not (0.0 < gamma <= 1.0):
        raise ValueError("gamma must lie in (0, 1]")
    if not (np.isfinite(beta) and beta >= 0.0):
        raise ValueError("beta must be finite and >= 0")
    B, K1, V = np.shape(logits_full)
    K = K1 - 1
    tokens = np.asarray(draft_tokens, np.int64).reshape(B, K)
    if mode == STOCHASTIC:
        probs = np.asarray(draft_probs, np.float32).astype(np.float64).reshape(B, K)
        unif = np.asarray(uniforms, np.float32).astype(np.float64).reshape(B, K1)
    elif mode != GREEDY:
        raise ValueError(f"unknown mode {mode}")
    res = Result(
        accept_len=np.full(B, -1, np.int64), next_token=np.full(B, -1, np.int64),
        flagged=np.zeros(B, bool), error=np.zeros(B, bool),
        lse=np.full((B, K1, 4), np.nan), D=np.full((B, K1), np.nan),
        gamma_eff=np.full((B, K1), np.nan), fused_argmax=np.full((B, K1), -1, np.int64),
        fused_gap_flag=np.zeros((B, K1), bool),
        candidate=np.full((B, K1), -1, np.int64), cand_flag=np.zeros((B, K1), bool),
        accept=np.zeros((B, K), bool), accept_margin=np.full((B, K), np.nan),
        logprobs=np.full((B, K1, V), np.nan) if want_logprobs else None)

    for bi in range(B):
        a_all = widen(logits_full[bi], dtype)
        b_all = widen(logits_comp[bi], dtype)
        t_all = widen(logits_ver[bi], dtype)
        # greedy decoding without a fused bonus never uses a and b of the bonus
        # row (Algorithm 1 emits argmax(t_{K+1})), so only used data is checked
        ab_rows = K if (mode == GREEDY and not fuse_bonus) else K1
        ok = bool(np.all(np.isfinite(a_all[:ab_rows])) and np.all(np.isfinite(b_all[:ab_rows]))
                  and np.all(np.isfinite(t_all)))
        ok = ok and bool(np.all((tokens[bi] >= 0) & (tokens[bi] < V)))
        if mode == STOCHASTIC:
            ok = ok and bool(np.all((probs[bi] > 0.0) & (probs[bi] <= 1.0)))
            ok = ok and bool(np.all((unif[bi] >= 0.0) & (unif[bi] < 1.0)))
        if not ok:
            res.error[bi] = True
            continue
        rows = []
        for k in range(K1):
            d = int(tokens[bi, k]) if k < K else None
            r = row_quantities(a_all[k], b_all[k], t_all[k], gamma, beta, divergence, lam, d,
                               delta_source)
            rows.append(r)
            res.lse[bi, k] = (r.lse_a, r.lse_b, r.lse_t, r.lse_s)
            res.D[bi, k] = r.D
            res.gamma_eff[bi, k] = r.gamma_eff
            if np.all(np.isfinite(r.s)):
                res.fused_argmax[bi, k] = argmax_first(r.s)
                res.fused_gap_flag[bi, k] = (top2_gap(r.s)
                                             < ARGMAX_BAND * max(1.0, abs(float(np.max(r.s)))))
            else:  # only in rows the step does not use: undefined, not compared
                res.fused_gap_flag[bi, k] = True
            if want_logprobs:
                res.logprobs[bi, k] = r.lq
        if mode == GREEDY:
            cand, cflag = greedy_candidates(rows, K, fuse_bonus)
            out = greedy_scan(rows, tokens[bi][None, :], K, fuse_bonus)
        else:
            cand, cflag = stochastic_candidates(rows, K, unif[bi, K])
            cand, cflag = cand[0], cflag[0]
            out = stochastic_scan(rows, tokens[bi][None, :], probs[bi][None, :],
                                  unif[bi][None, :], K)
        res.candidate[bi] = cand
        res.cand_flag[bi] = cflag
        res.accept_len[bi] = out[0][0]
        res.next_token[bi] = out[1][0]
        res.flagged[bi] = out[2][0]
        res.accept[bi] = out[3][0]
        res.accept_margin[bi] = out[4][0]
    return res


# ------------------------------------------------- cross-family vocabularies

def check_vocab_map(map_d, map_v, V_d: int, V_v: int):
    """The shared-token pairs as int64 arrays; raises ValueError unless they
    are two 1-D arrays of one length S >= 2, in range, each without repeats."""
    md = np.asarray(map_d, np.int64)
    mv = np.asarray(map_v, np.int64)
    if md.ndim != 1 or mv.shape != md.shape or md.size < 2:
        raise ValueError("map_d and map_v must be 1-D of one length S >= 2")
    if md.min() < 0 or md.max() >= V_d or mv.min() < 0 or mv.max() >= V_v:
        raise ValueError("a map entry lies outside its vocabulary")
    if np.unique(md).size != md.size or np.unique(mv).size != mv.size:
        raise ValueError("a vocabulary token appears in two pairs")
    return md, mv


def fuse_verify_xvocab(logits_full, logits_comp, logits_ver, map_d, map_v, draft_index,
                       draft_probs=None, uniforms=None, **kw) -> Result:
    """The step for a drafter and a verifier with different vocabularies
    (Section 4, "Cross-family portability"; appendix "Cross-family
    portability"): logits_full and logits_comp are [B, K+1, V_d] (drafter
    vocabulary), logits_ver [B, K+1, V_v] (verifier vocabulary), the S pairs
    (map_d[j], map_v[j]) the string-identical tokens, draft_index [B, K] pair
    indices in [0, S).  The rows are restricted to the pairs and the step runs
    on them unchanged; the emitted pair index j is committed as the verifier
    token map_v[j].  Returns fuse_verify's Result with next_token, candidate
    and fused_argmax as verifier tokens, the pair index of the next token in
    an extra field next_index, and logprobs (if asked for) over the pairs.
    """
    V_d = np.shape(logits_full)[-1]
    V_v = np.shape(logits_ver)[-1]
    md, mv = check_vocab_map(map_d, map_v, V_d, V_v)
    a = np.asarray(logits_full)[..., md]
    b = np.asarray(logits_comp)[..., md]
    t = np.asarray(logits_ver)[..., mv]
    res = fuse_verify(a, b, t, draft_index, draft_probs, uniforms, **kw)

    def to_verifier(j):
        j = np.asarray(j)
        return np.where(j >= 0, mv[np.maximum(j, 0)], -1)

    res.next_index = res.next_token.copy()
    res.next_token = to_verifier(res.next_token)
    res.candidate = to_verifier(res.candidate)
    res.fused_argmax = to_verifier(res.fused_argmax)
    return res


# ----------------------------------------------------------- the drafter's draw

@dataclass
class DraftResult:
    tokens: np.ndarray     # [rows] int, -1 on data error
    probs: np.ndarray      # [rows] softmax(a)[token], NaN on data error
    flagged: np.ndarray    # [rows] bool: the draw is a near-tie
    error: np.ndarray      # [rows] bool


def draft_sample(logits, uniforms=None, *, dtype=FP32, mode=GREEDY) -> DraftResult:
    """The augmented drafter's draw at each position (Section 3.2, item 1 of
    the three forward passes; the drafting line of Algorithm 1): from the
    drafter's full-context logits a, greedy decoding takes d = argmax a (the
    lowest index among ties) and sampling takes the inverse CDF of softmax(a)
    at the position's uniform u (index order, strict >).  Also returns the
    drafter's probability of its draw, softmax(a)[d], which the stochastic
    verification divides by.

    logits: [rows, V] in the stored dtype; uniforms: [rows] float32 (sampling
    only).  A row with a non-finite logit, or (sampling) a uniform outside
    [0, 1), is a data error.  Near-ties: an argmax whose top-2 gap is below
    ARGMAX_BAND * max(1, |top|), or an inverse-CDF target within CDF_BAND of
    a cumulative boundary, is flagged.
    """
    rows, V = np.shape(logits)
    out = DraftResult(tokens=np.full(rows, -1, np.int64), probs=np.full(rows, np.nan),
                      flagged=np.zeros(rows, bool), error=np.zeros(rows, bool))
    if mode == STOCHASTIC:
        unif = np.asarray(uniforms, np.float32).astype(np.float64).reshape(rows)
    elif mode != GREEDY:
        raise ValueError(f"unknown mode {mode}")
    for r in range(rows):
        a = widen(np.asarray(logits)[r], dtype)
        if not np.all(np.isfinite(a)) or (mode == STOCHASTIC and not 0.0 <= unif[r] < 1.0):
            out.error[r] = True
            continue
        la = log_softmax(a)
        if mode == GREEDY:
            d = argmax_first(a)
            out.flagged[r] = top2_gap(a) < ARGMAX_BAND * max(1.0, abs(float(a[d])))
        else:
            p = np.exp(la)
            idx, dist = inverse_cdf(p, unif[r])
            d = int(idx[0])
            out.flagged[r] = bool(dist[0] < CDF_BAND)
        out.tokens[r] = d
        out.probs[r] = float(np.exp(la[d]))
    return out
