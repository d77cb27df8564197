"""Hand-built edge cases (tests/golden/cases.json, written by make_golden.py from the oracle).

The CPU test checks that the oracle still produces the stored values; the GPU
test checks the CUDA path against them.  The inputs are small integers, so
the fused scores are exact in fp32 and the flagged cases here are exact ties,
which both sides must break toward the lowest index.
"""
import json
import os

import numpy as np
import pytest

import oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))
CASES = json.load(open(os.path.join(HERE, "golden", "cases.json")))["cases"]


def _inputs(c):
    i = c["inputs"]
    return (np.asarray(i["logits_full"], np.float32), np.asarray(i["logits_comp"], np.float32),
            np.asarray(i["logits_ver"], np.float32), np.asarray(i["draft_tokens"], np.int32),
            np.asarray(i["draft_probs"], np.float32), np.asarray(i["uniforms"], np.float32))


@pytest.mark.parametrize("c", CASES, ids=[c["name"] for c in CASES])
def test_oracle_reproduces_golden(c):
    a, b, t, d, p, u = _inputs(c)
    pr = c["params"]
    r = O.fuse_verify(a, b, t, d, p, u, dtype=O.FP32, gamma=pr["gamma"], beta=pr["beta"],
                      mode=pr["mode"], divergence=pr["divergence"],
                      fuse_bonus=bool(pr["fuse_bonus"]), want_logprobs=True)
    e = c["expected"]
    assert r.accept_len.tolist() == e["accept_len"]
    assert r.next_token.tolist() == e["next_token"]
    assert r.candidate.tolist() == e["candidate"]
    assert np.allclose(r.D, e["D"], atol=1e-13)
    assert np.allclose(r.logprobs, e["fused_logprobs"], atol=1e-13)


@pytest.mark.gpu
@pytest.mark.parametrize("c", CASES, ids=[c["name"] for c in CASES])
def test_gpu_matches_golden(c):
    import torch

    from paper_2608_26004_gb300 import asymspec as A
    a, b, t, d, p, u = _inputs(c)
    dev = "cuda"
    x = [torch.from_numpy(v).to(dev) for v in (a, b, t, d, p, u)]
    pr = c["params"]
    fv = A.FuseVerify(a.shape[0], a.shape[1] - 1)
    r = fv(*x, gamma=pr["gamma"], beta=pr["beta"], mode=pr["mode"], divergence=pr["divergence"],
           fuse_bonus=bool(pr["fuse_bonus"]), row_stats=True, row_tokens=True,
           fused_logprobs=True)
    torch.cuda.synchronize()
    e = c["expected"]
    assert r["accept_len"].cpu().tolist() == e["accept_len"]
    assert r["next_token"].cpu().tolist() == e["next_token"]
    rt = r["row_tokens"].cpu().numpy()
    assert rt[..., 0].tolist() == e["fused_argmax"]
    assert rt[..., 1].tolist() == e["candidate"]
    rs = r["row_stats"].cpu().numpy()
    assert np.allclose(rs[..., 4], e["D"], atol=1e-5)
    assert np.allclose(rs[..., 5], e["gamma_eff"], atol=1e-5)
    assert np.allclose(r["fused_logprobs"].cpu().numpy(), e["fused_logprobs"], atol=1e-5)
