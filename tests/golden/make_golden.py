"""Writes tests/golden/cases.json: small hand-built inputs and the oracle's outputs.

Only oracle/ computes the stored values.  Each case isolates one rule of the
step (cited in its "cites" field); the inputs are chosen by hand so the rule
decides the outcome with a wide margin.  Run from the repository root:

    python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle as O  # noqa: E402


def case(name, cites, a, b, t, d, probs=None, unif=None, mode=O.GREEDY, gamma=0.5, beta=1.0,
         div=O.DIV_JSD, fuse_bonus=False):
    a = np.asarray(a, np.float32)
    b = np.asarray(b, np.float32)
    t = np.asarray(t, np.float32)
    B, K1, V = a.shape
    d = np.asarray(d, np.int32).reshape(B, K1 - 1)
    probs = np.full((B, K1 - 1), 0.5, np.float32) if probs is None else np.asarray(probs, np.float32)
    unif = np.full((B, K1), 0.5, np.float32) if unif is None else np.asarray(unif, np.float32)
    r = O.fuse_verify(a, b, t, d, probs, unif, dtype=O.FP32, gamma=gamma, beta=beta, mode=mode,
                      divergence=div, fuse_bonus=fuse_bonus, want_logprobs=True)
    return {
        "name": name, "cites": cites,
        "params": {"mode": mode, "gamma": gamma, "beta": beta, "divergence": div,
                   "fuse_bonus": int(fuse_bonus)},
        "inputs": {"logits_full": a.tolist(), "logits_comp": b.tolist(), "logits_ver": t.tolist(),
                   "draft_tokens": d.tolist(), "draft_probs": probs.tolist(),
                   "uniforms": unif.tolist()},
        "expected": {"accept_len": r.accept_len.tolist(), "next_token": r.next_token.tolist(),
                     "flagged": r.flagged.tolist(), "D": r.D.tolist(),
                     "gamma_eff": r.gamma_eff.tolist(), "fused_argmax": r.fused_argmax.tolist(),
                     "candidate": r.candidate.tolist(), "accept": r.accept.tolist(),
                     "fused_logprobs": r.logprobs.tolist()},
    }


def main():
    cases = []
    # d_1 passes Eq. 4, d_2 fails; the first rejection emits the fused argmax,
    # which differs from the verifier's own argmax at that position.
    a = [[[0, 0, 3, 0, 0], [0, 4, 0, 0, 0], [0, 0, 0, 0, 1]]]
    b = [[[0, 0, 3, 0, 0], [0, 0, 0, 0, 0], [0, 0, 0, 0, 0]]]
    t = [[[0, 0, 3, 0, 0], [2.5, 0, 0, 0, 0], [0, 0, 0, 6, 0]]]
    cases.append(case("first_rejection_emits_fused_argmax", "Eq. 2, Eq. 4, Algorithm 1",
                      a, b, t, [[2, 4]]))
    # every draft passes: the bonus position emits argmax(t_K) (unfused) ...
    a = [[[0, 0, 4, 0], [0, 4, 0, 0], [9, 0, 0, 0]]]
    b = [[[0, 0, 4, 0], [0, 4, 0, 0], [0, 0, 0, 0]]]
    t = [[[0, 0, 4, 0], [0, 4, 0, 0], [0, 0, 5, 0]]]
    cases.append(case("all_accepted_bonus_is_verifier_argmax",
                      "Algorithm 1 (emission after the loop)", a, b, t, [[2, 1]]))
    # ... or the fused argmax when the bonus is fused
    cases.append(case("all_accepted_fused_bonus", "Fig. 1 caption reading of the bonus",
                      a, b, t, [[2, 1]], fuse_bonus=True))
    # an exact tie in the fused scores resolves to the lowest index
    a = [[[0, 1, 0, 1, 0, 0], [0, 0, 0, 0, 0, 0]]]
    b = [[[0, 0, 0, 0, 0, 0], [0, 0, 0, 0, 0, 0]]]
    t = [[[0, 2, 0, 2, 0, 3], [0, 0, 0, 0, 0, 0]]]
    cases.append(case("fused_tie_lowest_index", "Eq. 2 (argmax)", a, b, t, [[0]]))
    # beta = 0 and gamma = 1: the plain verifier argmax is emitted at a rejection
    a = [[[3, 0, 0], [0, 0, 0]]]
    b = [[[0, 3, 0], [0, 0, 0]]]
    t = [[[0, 0, 2], [0, 1, 0]]]
    cases.append(case("beta0_gamma1", "Section 3.3 (degenerate case)", a, b, t, [[0]],
                      gamma=1.0, beta=0.0))
    # identical contexts: delta = 0, D = 0, gamma_eff = gamma
    a = [[[1, 2, 3, 0.5], [0, 1, 0, 2], [2, 2, 0, 1]]]
    cases.append(case("identical_contexts", "Eq. 1, Eq. 3, Appendix A (gamma_eff(0) = gamma)",
                      a, a, [[[0, 1, 1, 0], [3, 0, 0, 0], [0, 0, 0, 1]]], [[2, 3]]))
    # nearly disjoint supports: D -> ln 2, gamma_eff -> gamma / 2
    a = [[[30, -30], [0, 0]]]
    b = [[[-30, 30], [0, 0]]]
    t = [[[0, 0], [0, 0]]]
    cases.append(case("near_disjoint_supports", "Eq. 3 and Appendix A (JSD <= ln 2)",
                      a, b, t, [[0]]))
    # stochastic: the draft is rejected (u close to 1) and the residual is sampled
    a = [[[2, 0, 0, 0], [0, 0, 0, 0]]]
    b = [[[0, 0, 0, 0], [0, 0, 0, 0]]]
    t = [[[-2, 0, 1, 0], [0, 0, 0, 0]]]
    pa = np.exp(np.float64(2)) / (np.exp(np.float64(2)) + 3)
    cases.append(case("stochastic_rejection_residual_draw",
                      "speculative sampling residual (extension)", a, b, t, [[0]],
                      probs=[[pa]], unif=[[0.95, 0.3]], mode=O.STOCHASTIC))
    cases.append(case("stochastic_bonus_draw", "speculative sampling (extension)", a, a,
                      [[[2, 0, 0, 0], [0, 1, 2, 3]]], [[0]], probs=[[pa]],
                      unif=[[0.1, 0.7]], mode=O.STOCHASTIC, gamma=1.0))
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "cases.json")
    with open(path, "w") as f:
        json.dump({"generator": "tests/golden/make_golden.py (oracle/ only)", "cases": cases},
                  f, indent=1)
    print(f"wrote {len(cases)} cases to {path}")


if __name__ == "__main__":
    main()
