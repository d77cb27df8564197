"""Shared helpers of the GPU parity tests: run the C ABI, compare with the oracle."""
from __future__ import annotations

import numpy as np

import oracle as O
from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth

LOGPROB_TOL = {synth.FP32: 1e-5, synth.BF16: 2e-3}
LSE_TOL = 2e-5
D_TOL = 1e-5
GAMMA_TOL = 1e-5


def device_inputs(batch, torch, device="cuda"):
    """Host arrays of a synth.Batch (or an equivalent object) as CUDA tensors."""
    def logits(x):
        if batch.dtype == synth.BF16:
            t = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16)
        else:
            t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
        return t.to(device)
    return dict(
        a=logits(batch.logits_full), b=logits(batch.logits_comp), t=logits(batch.logits_ver),
        tokens=torch.from_numpy(np.ascontiguousarray(batch.draft_tokens, np.int32)).to(device),
        probs=torch.from_numpy(np.ascontiguousarray(batch.draft_probs, np.float32)).to(device),
        unif=torch.from_numpy(np.ascontiguousarray(batch.uniforms, np.float32)).to(device))


def run_gpu(batch, torch, *, mode, divergence=A.DIV_JSD, gamma=0.5, beta=1.0, lam=0.1,
            fuse_bonus=False, cluster_size=0, logprobs=True, inputs=None, kernel=0, full=True,
            delta_source=A.DELTA_AB, tokens=True, block_threads=0):
    """One call of asymspec_fuse_verify_ex through the binding; numpy results.

    full=True asks for every debug output (row statistics, fused log-probs),
    which runs the full per-row program; full=False asks only for the row
    tokens (tokens=True) or for nothing but the accepted lengths and next
    tokens (tokens=False: the production program the benchmark times).
    """
    if full == "row":  # the production program's outputs only
        full, tokens = False, False
    x = inputs if inputs is not None else device_inputs(batch, torch)
    elt = 4 if batch.dtype == synth.FP32 else 2
    if kernel == A.KERNEL_TMA and (batch.V * elt) % 16:
        kernel = A.KERNEL_AUTO  # rows not 16-byte aligned: only the generic kernel applies
    fv = A.FuseVerify(batch.B, batch.K)
    res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], gamma=gamma, beta=beta,
             lam=lam, mode=mode, divergence=divergence, fuse_bonus=fuse_bonus,
             row_stats=full, row_tokens=full or tokens, fused_logprobs=full and logprobs,
             cluster_size=cluster_size, kernel=kernel, delta_source=delta_source,
             block_threads=block_threads)
    torch.cuda.synchronize()
    out = {k: v.cpu().numpy() for k, v in res.items()}
    out["workspace_after"] = fv.workspace.cpu().numpy()
    return out


def run_oracle(batch, *, mode, divergence=A.DIV_JSD, gamma=0.5, beta=1.0, lam=0.1,
               fuse_bonus=False, logprobs=True, select=None, delta_source=A.DELTA_AB):
    """The oracle on the batch (or the selected elements); the result carries
    the parameters the validity checks of compare() need."""
    sel = slice(None) if select is None else select
    o = O.fuse_verify(batch.logits_full[sel], batch.logits_comp[sel], batch.logits_ver[sel],
                      batch.draft_tokens[sel], batch.draft_probs[sel], batch.uniforms[sel],
                      dtype=batch.dtype, gamma=gamma, beta=beta, mode=mode,
                      divergence=divergence, lam=lam, fuse_bonus=fuse_bonus,
                      want_logprobs=logprobs, delta_source=delta_source)
    o.params = dict(beta=beta, fuse_bonus=fuse_bonus, delta_source=delta_source)
    return o


# ------------------------------------------------- validity of near-tie decisions

def _row(batch, bi, k, params):
    a = O.widen(batch.logits_full[bi, k], batch.dtype)
    b = O.widen(batch.logits_comp[bi, k], batch.dtype)
    t = O.widen(batch.logits_ver[bi, k], batch.dtype)
    return O.row_quantities(a, b, t, 0.5, params["beta"], O.DIV_NONE,
                            delta_source=params["delta_source"])


def token_valid(batch, bi, k, token, mode, params) -> bool:
    """Whether `token`, emitted by a stop at row k of batch element bi, is a
    correct emission within the near-tie bands: greedy, its score lies within
    ARGMAX_BAND * max(1, |top|) of the row's maximum (fused scores, or the
    verifier's logits on an unfused bonus row); stochastic, it has positive
    mass under the row's sampled distribution (the residual on draft rows, the
    fused target when that residual is below CDF_BAND in total or on the bonus
    row) and its cumulative interval [C(y-1), C(y)) lies within CDF_BAND of
    the target u_K * total (float64, exact inputs)."""
    K, V = batch.K, batch.V
    if not 0 <= token < V:
        return False
    r = _row(batch, bi, k, params)
    if mode == A.MODE_GREEDY:
        z = r.s if (k < K or params["fuse_bonus"]) else r.t
        top = float(np.max(z))
        return bool(z[token] >= top - O.ARGMAX_BAND * max(1.0, abs(top)))
    q = np.exp(r.lq)
    u = float(np.float32(batch.uniforms[bi, K]))
    masses = [q]
    if k < K:
        resid = np.maximum(q - np.exp(r.la), 0.0)
        R = float(np.sum(resid))
        masses = [resid] if R >= O.CDF_BAND else ([resid, q] if R > 0.0 else [q])
    for m in masses:
        if not m[token] > 0.0:
            continue
        cum = np.cumsum(m)
        lo = float(cum[token - 1]) if token > 0 else 0.0
        tau = u * float(cum[-1])
        if lo - O.CDF_BAND <= tau < float(cum[token]) + O.CDF_BAND:
            return True
    return False


def argmax_valid(batch, bi, k, token, params) -> bool:
    """The fused argmax of row k: within ARGMAX_BAND of the maximum of s."""
    if not 0 <= token < batch.V:
        return False
    s = _row(batch, bi, k, params).s
    top = float(np.max(s))
    return bool(s[token] >= top - O.ARGMAX_BAND * max(1.0, abs(top)))


def check_decisions(batch, sel, L, N, o, mode):
    """accept_len / next_token of every batch element against the oracle.

    Elements the oracle does not flag: bit-exact.  Flagged elements: every
    acceptance decision the GPU's scan reached agrees with the oracle's
    unless its margin lies within ACCEPT_BAND, and the emitted token is a
    correct emission at the row where the GPU's scan stopped (token_valid).
    Returns the number of flagged elements (data errors excluded)."""
    params = getattr(o, "params", dict(beta=1.0, fuse_bonus=False, delta_source=A.DELTA_AB))
    K = batch.K
    err = o.error
    ok = ~o.flagged & ~err
    bad = np.nonzero(ok & ((L != o.accept_len) | (N != o.next_token)))[0]
    assert bad.size == 0, (
        f"accept/next mismatch at b={sel[bad][:8]}: gpu {L[bad][:8]} {N[bad][:8]} "
        f"oracle {o.accept_len[bad][:8]} {o.next_token[bad][:8]}")
    for i in np.nonzero(o.flagged & ~err)[0]:
        lg = int(L[i])
        assert 0 <= lg <= K, f"b={sel[i]}: accepted length {lg} out of range"
        for j in range(min(lg, K - 1) + 1 if lg < K else K):
            gpu_acc = j < lg
            assert gpu_acc == bool(o.accept[i, j]) or abs(o.accept_margin[i, j]) < O.ACCEPT_BAND, \
                f"b={sel[i]}: decision {j} differs outside the near-tie band"
        assert token_valid(batch, sel[i], lg, int(N[i]), mode, params), \
            f"b={sel[i]}: flagged element emits {int(N[i])} at row {lg}, not a valid emission"
    return int((o.flagged & ~err).sum())


def compare(batch, g, o, *, mode, select=None, logprobs=True, check_stats=True,
            max_flagged=None):
    """Asserts GPU == oracle within the stated tolerances; returns counters.

    accept_len / next_token: bit-exact except batch elements the oracle flags
    as reaching a near-tie, which are checked for validity instead
    (check_decisions).  Per-row decisions and tokens: exact except rows whose
    own decision is a near-tie, checked for validity.  Fused log-probs: max
    |error| within 2e-3 (bf16 inputs) or 1e-5 (fp32 inputs).  max_flagged: a
    ceiling on the fraction of (non-error) elements the oracle flags.
    """
    sel = np.arange(batch.B) if select is None else np.asarray(select)
    L, N = g["accept_len"][sel], g["next_token"][sel]
    err = o.error
    assert np.array_equal(L < 0, err), "data-error elements differ"
    assert np.array_equal(N < 0, err)
    ok = ~o.flagged & ~err
    nflag = check_decisions(batch, sel, L, N, o, mode)
    params = getattr(o, "params", dict(beta=1.0, fuse_bonus=False, delta_source=A.DELTA_AB))
    K1 = batch.K + 1
    good = ~err
    if "row_tokens" not in g:  # the production program: accept_len / next_token only
        ngood = int(good.sum())
        frac = nflag / ngood if ngood else 0.0
        if max_flagged is not None:
            assert frac <= max_flagged, f"{nflag} of {ngood} elements flagged ({frac:.1%})"
        return dict(compared=int(ok.sum()), flagged=nflag, flagged_frac=frac,
                    errors=int(err.sum()), logprob_err=None, rows=int(len(sel) * K1))
    rt = g["row_tokens"][sel]
    # fused argmax: compared wherever the GPU computed it (-1 = not needed by
    # the production program, only the greedy bonus row); draft rows always
    # have it.  Near-ties: a valid argmax within the band.
    computed = rt[..., 0] >= 0
    assert np.all(computed[good][:, :batch.K]), "fused argmax missing on draft rows"
    fa_ok = good[:, None] & ~o.fused_gap_flag & computed
    assert np.array_equal(rt[..., 0][fa_ok], o.fused_argmax[fa_ok]), "fused argmax differs"
    # (rows whose fused scores are not all finite, which the step does not
    # use, have no defined argmax: the oracle reports -1 there)
    for i, k in np.argwhere(good[:, None] & o.fused_gap_flag & computed & (o.fused_argmax >= 0)):
        assert argmax_valid(batch, sel[i], k, int(rt[i, k, 0]), params), \
            f"fused argmax of b={sel[i]} row {k} is not within the near-tie band"
    # the token each row would emit: exact, or valid where the row's own
    # decision is a near-tie
    c_ok = good[:, None] & ~o.cand_flag
    cbad = np.argwhere(c_ok & (rt[..., 1] != o.candidate))
    assert cbad.size == 0, f"row candidates differ at {cbad[:6]}"
    for i, k in np.argwhere(good[:, None] & o.cand_flag):
        assert token_valid(batch, sel[i], k, int(rt[i, k, 1]), mode, params), \
            f"row candidate of b={sel[i]} row {k} is not a valid emission"
    if "row_stats" in g:
        rs = g["row_stats"][sel]
        acc_gpu = rs[:, :batch.K, 6] < 0
        m_ok = good[:, None] & (np.abs(o.accept_margin) >= O.ACCEPT_BAND)
        abad = np.argwhere(m_ok & (acc_gpu != o.accept))
        assert abad.size == 0, f"acceptance decisions differ at {abad[:6]}"
    if check_stats and "row_stats" in g and good.any():
        gl = rs[good][..., :4]
        ol = o.lse[good]
        diff = np.abs(gl - ol)
        assert np.nanmax(diff) <= LSE_TOL * max(1.0, float(np.max(np.abs(ol)))), \
            f"LSE error {np.nanmax(diff)}"
        dD = np.abs(rs[good][..., 4] - o.D[good])
        assert np.max(dD) <= D_TOL, f"D error {np.max(dD)}"
        dg = np.abs(rs[good][..., 5] - o.gamma_eff[good])
        assert np.max(dg) <= GAMMA_TOL, f"gamma_eff error {np.max(dg)}"
    lp_err = None
    if logprobs and o.logprobs is not None and "fused_logprobs" in g:
        glp = g["fused_logprobs"][sel][good]
        lp_err = float(np.max(np.abs(glp - o.logprobs[good]))) if good.any() else 0.0
        assert lp_err <= LOGPROB_TOL[batch.dtype], f"fused log-prob error {lp_err}"
    # the per-element tickets (after the 256-byte aligned row records) return to zero
    rec_bytes = -(-batch.B * K1 * 16 // 256) * 256
    tickets = g["workspace_after"][rec_bytes:rec_bytes + 4 * batch.B]
    assert np.all(tickets == 0), "tickets not left zeroed"
    ngood = int(good.sum())
    frac = nflag / ngood if ngood else 0.0
    if max_flagged is not None:
        assert frac <= max_flagged, f"{nflag} of {ngood} elements flagged ({frac:.1%})"
    return dict(compared=int(ok.sum()), flagged=nflag, flagged_frac=frac,
                errors=int(err.sum()), logprob_err=lp_err, rows=int(len(sel) * K1))
