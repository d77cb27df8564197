"""The drafter's draw on the GPU (asymspec_draft_sample) against the oracle.

Greedy tokens are compared exactly on every row (the argmax of the stored
values is exact on both sides).  Sampled tokens are compared exactly where
the oracle does not flag the target as within CDF_BAND of a cumulative
boundary; on flagged rows the GPU's token must still be a valid draw near the
target.  Probabilities agree within PROB_RTOL: the kernel forms
softmax(a)[d] in fp32 from ex2 of fma-rounded exponents (relative error below
1e-5 for |logit| <= 100) over per-thread sums of at most ~600 terms (below
4e-5), so 1e-4 bounds the two together.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth

pytestmark = pytest.mark.gpu

GREEDY, STOCH = A.MODE_GREEDY, A.MODE_STOCHASTIC
PROB_RTOL = 1e-4
BF16_NAN, BF16_PINF, BF16_NINF = 0x7FC0, 0x7F80, 0xFF80


@pytest.fixture(scope="module")
def torch():
    import torch as _torch
    assert _torch.cuda.is_available(), "the gpu tests need a CUDA device"
    from paper_2608_26004_gb300 import build
    build.build_cuda()
    A.lib()
    return _torch


def to_device(torch, logits, dtype, offset=0):
    """[rows, V] host logits (uint16 bit patterns for bf16) as a CUDA tensor,
    optionally starting `offset` elements into a larger allocation."""
    rows, V = logits.shape
    flat = np.ascontiguousarray(logits).reshape(-1)
    if dtype == synth.BF16:
        t = torch.from_numpy(flat.view(np.int16).copy()).view(torch.bfloat16)
    else:
        t = torch.from_numpy(flat.astype(np.float32))
    if offset:
        t = torch.cat([torch.zeros(offset, dtype=t.dtype), t])
    t = t.cuda()
    return t[offset:].view(rows, V)


def run(torch, logits, dtype, mode, unif=None, offset=0, cluster_size=0):
    a = to_device(torch, logits, dtype, offset)
    u = torch.from_numpy(np.asarray(unif, np.float32)).cuda() if unif is not None else None
    tok, pr = A.draft_tokens(a, u, mode=mode, cluster_size=cluster_size)
    torch.cuda.synchronize()
    return tok.cpu().numpy(), pr.cpu().numpy()


def check_valid_draw(logits, dtype, u, tok):
    """A flagged sampled row: the token has positive mass and its cumulative
    interval lies within 2 CDF_BAND of the target."""
    a = O.widen(logits, dtype)
    p = np.exp(O.log_softmax(a))
    assert 0 <= tok < p.size and p[tok] > 0
    cum = np.cumsum(p)
    lo = cum[tok - 1] if tok > 0 else 0.0
    assert lo - 2 * O.CDF_BAND <= u < cum[tok] + 2 * O.CDF_BAND or tok == np.nonzero(p)[0][-1]


def compare(logits, dtype, mode, unif, tok, pr):
    o = O.draft_sample(logits, unif, dtype=dtype, mode=mode)
    err = o.error
    assert np.array_equal(tok[err], np.full(err.sum(), -1)), "error rows must give token -1"
    assert np.all(np.isnan(pr[err]))
    good = ~err
    if mode == GREEDY:
        assert np.array_equal(tok[good], o.tokens[good])
    else:
        same = good & ~o.flagged
        assert np.array_equal(tok[same], o.tokens[same])
        for r in np.nonzero(good & o.flagged)[0]:
            check_valid_draw(logits[r], dtype, float(unif[r]), int(tok[r]))
    # the probability of the GPU's own token (equal to the oracle's where the tokens agree)
    for r in np.nonzero(good)[0]:
        lp = O.log_softmax(O.widen(logits[r], dtype))
        np.testing.assert_allclose(pr[r], np.exp(lp[tok[r]]), rtol=PROB_RTOL, atol=1e-30)
    return o


def rows_of(batch):
    return batch.logits_full.reshape(-1, batch.V), batch.uniforms.reshape(-1)


SIZES = [
    # rows-producing (B, K), V, dtype               path
    ((3, 3), 1000, synth.FP32),    # float4 vectors, 250 per row: one partial round
    ((2, 2), 4099, synth.BF16),    # odd V: scalar path, ragged tail
    ((4, 1), 8200, synth.BF16),    # 1025 uint4 per row: 4 full rounds + 1 vector
    ((2, 3), 32000, synth.FP32),   # 8000 float4: unrolled batches and a tail
    ((1, 3), 151936, synth.BF16),  # a Qwen3-sized row
    ((1, 2), 151937, synth.FP32),  # scalar path, 594 elements per thread
]


@pytest.mark.parametrize("cluster", [0, 1, 8], ids=["auto", "C1", "C8"])
@pytest.mark.parametrize("mode", [GREEDY, STOCH], ids=["greedy", "stochastic"])
@pytest.mark.parametrize("size", SIZES, ids=[f"V{v}_{'bf16' if d else 'fp32'}" for _, v, d in SIZES])
def test_draft_matches_oracle(torch, size, mode, cluster):
    # C CTAs split each row into C slices (auto: 8 for these few rows)
    (B, K), V, dtype = size
    batch = synth.generate(synth.Recipe(), 0xD7A0 + V, B, K, V, dtype)
    logits, unif = rows_of(batch)
    tok, pr = run(torch, logits, dtype, mode, unif, cluster_size=cluster)
    compare(logits, dtype, mode, unif, tok, pr)


@pytest.mark.parametrize("mode", [GREEDY, STOCH], ids=["greedy", "stochastic"])
def test_draft_cluster_sizes_agree(torch, mode):
    # every cluster size, including slices that end inside a round (160 fp32:
    # 40 vectors, slices of 5) and empty trailing slices (9 bf16 on the scalar
    # path: C = 8 gives slices of 2 and leaves the last three empty)
    for (B, K), V, dtype in (((4, 3), 8200, synth.BF16), ((2, 1), 160, synth.FP32),
                             ((2, 1), 9, synth.BF16)):
        batch = synth.generate(synth.Recipe(), 0xD7C0 + V, B, K, V, dtype)
        logits, unif = rows_of(batch)
        for c in (1, 2, 4, 8):
            tok, pr = run(torch, logits, dtype, mode, unif, cluster_size=c)
            compare(logits, dtype, mode, unif, tok, pr)


@pytest.mark.parametrize("dtype", [synth.FP32, synth.BF16], ids=["fp32", "bf16"])
@pytest.mark.parametrize("spike", [75.0, 90.0, 120.0])
def test_draft_entry_far_above_its_warp_reference(torch, dtype, spike):
    # one entry `spike` nats above the rest, outside the first round of any
    # warp: its group's mass reaches 2^100 (or overflows) against the warp's
    # first-round reference, and the CTA redoes its slice against the slice
    # maximum; the other rows keep the one-pass result
    V = 16384
    rng = np.random.default_rng(5)
    rows = (rng.standard_normal((4, V)) * 2.0).astype(np.float32)
    rows[0, 9000] = spike
    rows[1, 15000] = spike / 2
    rows[2, 5000], rows[2, 12000] = spike, spike - 1.0
    host = rows if dtype == synth.FP32 else (rows.view(np.uint32) >> 16).astype(np.uint16)
    unif = np.array([0.5, 0.3, 0.9, 0.7], np.float32)
    for c in (1, 2, 8):
        for mode in (GREEDY, STOCH):
            tok, pr = run(torch, host, dtype, mode, unif, cluster_size=c)
            compare(host, dtype, mode, unif, tok, pr)
            assert tok[0] == 9000


@pytest.mark.parametrize("mode", [GREEDY, STOCH], ids=["greedy", "stochastic"])
def test_draft_zipf_profile_full_batch(torch, mode):
    # every drafter row of a B=64, K=7, V=128256 bf16 step (Zipf-shaped
    # logits): 512 rows, the launch a full step's drafting would make at once
    w = synth.CONFIGS[2]
    batch = synth.make_config(2)
    logits, unif = rows_of(batch)
    assert logits.shape == (w.B * (w.K + 1), w.V)
    tok, pr = run(torch, logits, w.dtype, mode, unif)
    o = compare(logits, w.dtype, mode, unif, tok, pr)
    assert not o.error.any()


@pytest.mark.parametrize("dtype", [synth.FP32, synth.BF16], ids=["fp32", "bf16"])
def test_draft_ties_lowest_index(torch, dtype):
    V = 4096
    rows = np.zeros((5, V), np.float32)
    rows[0, [7, 3000, 4095]] = 5.0      # across threads: the lowest index
    rows[1, [17, 18, 19]] = 2.0         # inside one vector
    rows[2, :] = 1.0                    # every entry ties: index 0
    rows[3, [2048 + 5, 5]] = 3.0        # same thread and lane slot, later round second
    rows[4, [4095]] = 1e-3              # the last entry alone
    host = rows if dtype == synth.FP32 else (rows.view(np.uint32) >> 16).astype(np.uint16)
    tok, pr = run(torch, host, dtype, GREEDY)
    assert list(tok) == [7, 17, 0, 5, 4095]
    compare(host, dtype, GREEDY, None, tok, pr)


@pytest.mark.parametrize("dtype", [synth.FP32, synth.BF16], ids=["fp32", "bf16"])
def test_draft_data_errors_only_touch_their_rows(torch, dtype):
    V = 2000
    batch = synth.generate(synth.Recipe(), 0xD7E0, 2, 3, V, dtype)
    logits, unif = rows_of(batch)
    logits = logits.copy()
    unif = unif.copy()
    if dtype == synth.FP32:
        logits[1, 100], logits[3, 1999], logits[5, 0] = np.nan, np.inf, -np.inf
    else:
        logits[1, 100], logits[3, 1999], logits[5, 0] = BF16_NAN, BF16_PINF, BF16_NINF
    unif[6], unif[7] = 1.0, np.nan
    for mode in (GREEDY, STOCH):
        tok, pr = run(torch, logits, dtype, mode, unif)
        o = compare(logits, dtype, mode, unif, tok, pr)
        bad = {1, 3, 5} | ({6, 7} if mode == STOCH else set())
        assert set(np.nonzero(o.error)[0]) == bad
        assert set(np.nonzero(tok < 0)[0]) == bad


def test_draft_boundaries_and_smallest_vocabulary(torch):
    # V = 2 (scalar path); u = 0 takes the first entry of positive mass;
    # u just below 1 the last
    logits = np.array([[0.0, 0.0], [-200.0, 0.0], [0.0, 1.0], [3.0, -3.0]], np.float32)
    unif = np.array([0.0, 0.0, np.float32(1.0) - np.float32(2**-24), 0.49], np.float32)
    tok, pr = run(torch, logits, synth.FP32, STOCH, unif)
    compare(logits, synth.FP32, STOCH, unif, tok, pr)
    assert tok[0] == 0 and tok[2] == 1
    assert tok[1] == 1  # e^-200 is below the fp32 range: no mass
    tok, pr = run(torch, logits, synth.FP32, GREEDY)
    assert list(tok) == [0, 1, 1, 0]


@pytest.mark.parametrize("dtype", [synth.FP32, synth.BF16], ids=["fp32", "bf16"])
def test_draft_unaligned_rows_take_the_scalar_path(torch, dtype):
    # logits starting one element past a 16-byte boundary: same results
    V = 3072
    batch = synth.generate(synth.Recipe(), 0xD7B0, 2, 2, V, dtype)
    logits, unif = rows_of(batch)
    for mode in (GREEDY, STOCH):
        t0, p0 = run(torch, logits, dtype, mode, unif)
        t1, p1 = run(torch, logits, dtype, mode, unif, offset=1)
        compare(logits, dtype, mode, unif, t1, p1)
        assert np.array_equal(t0, t1)
        np.testing.assert_allclose(p0, p1, rtol=PROB_RTOL)


def test_draft_stratified_uniforms_reproduce_the_distribution(torch):
    # u_i = (i + 1/2) / N: each token is drawn N p_j times up to one, for
    # the inverse CDF of any distribution (a property at any N)
    V, N = 50, 4096
    rng = np.random.default_rng(11)
    a = (rng.standard_normal(V) * 1.5).astype(np.float32)
    logits = np.repeat(a[None, :], N, axis=0)
    unif = ((np.arange(N) + 0.5) / N).astype(np.float32)
    tok, _ = run(torch, logits, synth.FP32, STOCH, unif)
    p = np.exp(O.log_softmax(a.astype(np.float64)))
    counts = np.bincount(tok, minlength=V)
    assert np.all(np.abs(counts - N * p) <= 1.01)  # boundaries move by fp32 rounding only
    assert np.all(np.diff(tok) >= 0)  # monotone in u


def test_draft_no_rows_is_a_no_op(torch):
    a = torch.zeros((0, 64), dtype=torch.float32, device="cuda")
    tok, pr = A.draft_tokens(a)
    assert tok.numel() == 0 and pr.numel() == 0
