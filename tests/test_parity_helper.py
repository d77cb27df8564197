"""The near-tie validity checks of the GPU parity helper, on the CPU.

check_decisions and token_valid decide whether a GPU result that differs
from the oracle's on a flagged (near-tie) batch element is still a correct
emission.  Here they are fed the oracle's own results, which must pass, and
results with a planted mistake (a wrong token, a wrong accepted length),
which must fail.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth
from tests._parity import argmax_valid, check_decisions, run_oracle, token_valid


def _batch(mode_seed):
    return synth.generate(synth.Recipe(sigma_c=2.0, frac_lo=0.1, frac_hi=0.3), 500 + mode_seed,
                          6, 3, 3000, synth.FP32)


@pytest.mark.parametrize("mode", [A.MODE_GREEDY, A.MODE_STOCHASTIC])
def test_oracle_results_are_valid_emissions(mode):
    batch = _batch(mode)
    o = run_oracle(batch, mode=mode, logprobs=False)
    for b in range(batch.B):
        assert token_valid(batch, b, int(o.accept_len[b]), int(o.next_token[b]), mode, o.params)
        for k in range(batch.K + 1):
            assert token_valid(batch, b, k, int(o.candidate[b, k]), mode, o.params)
            assert argmax_valid(batch, b, k, int(o.fused_argmax[b, k]), o.params)
    # every element treated as flagged: the validity path accepts the oracle's own results
    o.flagged[:] = True
    assert check_decisions(batch, np.arange(batch.B), o.accept_len, o.next_token, o, mode) \
        == batch.B


def test_planted_wrong_tokens_are_rejected():
    batch = _batch(7)
    for mode in (A.MODE_GREEDY, A.MODE_STOCHASTIC):
        o = run_oracle(batch, mode=mode, logprobs=False)
        for b in range(batch.B):
            k, y = int(o.accept_len[b]), int(o.next_token[b])
            r = O.row_quantities(*(O.widen(x[b, k], batch.dtype) for x in
                                   (batch.logits_full, batch.logits_comp, batch.logits_ver)),
                                 0.5, 1.0, O.DIV_NONE)
            if mode == A.MODE_GREEDY:
                z = r.s if k < batch.K else r.t
                wrong = int(np.argmin(z))                      # the lowest score
            else:
                q = np.exp(r.lq)
                m = np.maximum(q - np.exp(r.la), 0.0) if k < batch.K else q
                if k < batch.K and m.sum() <= 0.0:
                    m = q
                cum = np.cumsum(m)
                # a token with mass whose interval lies far from the target
                tau = float(np.float32(batch.uniforms[b, batch.K])) * cum[-1]
                far = np.nonzero((m > 0) & (np.abs(cum - tau) > 0.05 * cum[-1]) &
                                 (np.abs(cum - m - tau) > 0.05 * cum[-1]))[0]
                wrong = int(far[0])
            assert not token_valid(batch, b, k, wrong, mode, o.params)
            assert not token_valid(batch, b, k, batch.V, mode, o.params)    # out of range


def test_planted_wrong_lengths_are_rejected():
    batch = _batch(9)
    o = run_oracle(batch, mode=A.MODE_STOCHASTIC, logprobs=False)
    o.flagged[:] = True
    sel = np.arange(batch.B)
    # an element whose decisions are all clear of the near-tie band
    b = int(np.nonzero(np.min(np.abs(o.accept_margin), axis=1) > 1e-3)[0][0])
    L = o.accept_len.copy()
    L[b] = (L[b] + 1) % (batch.K + 1)
    with pytest.raises(AssertionError):
        check_decisions(batch, sel, L, o.next_token, o, A.MODE_STOCHASTIC)
    L = o.accept_len.copy()
    with pytest.raises(AssertionError):   # unflagged: bit-exact required
        o2 = run_oracle(batch, mode=A.MODE_STOCHASTIC, logprobs=False)
        N = o2.next_token.copy()
        N[b] = (N[b] + 1) % batch.V
        check_decisions(batch, sel, L, N, o2, A.MODE_STOCHASTIC)
