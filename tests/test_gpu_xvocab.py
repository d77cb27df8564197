"""The cross-family step on the GPU (asymspec_fuse_verify_xvocab,
asymspec_xvocab_gather) against the oracle's fuse_verify_xvocab.

Drafter and verifier tokenise differently and share S tokens (Section 4,
"Cross-family portability"): the step runs over the rows restricted to the
pairs, and the emitted pair is committed as its verifier token.  The gather
is compared bit for bit with numpy indexing; accepted lengths, emitted pair
indices and verifier tokens exactly, except batch elements the oracle flags
as reaching a near-tie (its float64 decision lies within the bands of the
oracle's header).
"""
import functools

import numpy as np
import pytest

import oracle as O
from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth

pytestmark = pytest.mark.gpu

GREEDY, STOCH = A.MODE_GREEDY, A.MODE_STOCHASTIC


@pytest.fixture(scope="module")
def torch():
    import torch as _torch
    assert _torch.cuda.is_available(), "the gpu tests need a CUDA device"
    from paper_2608_26004_gb300 import build
    build.build_cuda()
    A.lib()
    return _torch


def dev(torch, x, dtype=None):
    x = np.ascontiguousarray(x)
    if dtype == synth.BF16:
        return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(x).cuda()


def run(torch, x, mode, *, gamma=0.5, beta=1.0, map_d=None, map_v=None, draft=None,
        calls=1):
    """One (or `calls`) asymspec_fuse_verify_xvocab on a synth.XBatch; numpy results."""
    md = dev(torch, np.asarray(x.map_d if map_d is None else map_d, np.int32))
    mv = dev(torch, np.asarray(x.map_v if map_v is None else map_v, np.int32))
    a, b = dev(torch, x.logits_full, x.dtype), dev(torch, x.logits_comp, x.dtype)
    t = dev(torch, x.logits_ver, x.dtype)
    d = dev(torch, np.asarray(x.draft_tokens if draft is None else draft, np.int32))
    pr, u = dev(torch, x.draft_probs.astype(np.float32)), dev(torch, x.uniforms.astype(np.float32))
    nbytes = A.xvocab_workspace_bytes(x.B, x.K, x.S, x.V_d, x.V_v, x.dtype)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    L = torch.empty(x.B, dtype=torch.int32, device="cuda")
    N = torch.empty_like(L)
    idx = torch.empty_like(L)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    gate = A.gate_params(gamma=gamma, beta=beta, mode=mode)
    stream = torch.cuda.current_stream().cuda_stream
    outs = []
    for _ in range(calls):
        st = A.fuse_verify_xvocab(a.data_ptr(), b.data_ptr(), x.V_d, t.data_ptr(), x.V_v,
                                  md.data_ptr(), mv.data_ptr(), x.S, d.data_ptr(),
                                  pr.data_ptr(), u.data_ptr(), x.B, x.K, x.dtype, gate,
                                  L.data_ptr(), N.data_ptr(), idx.data_ptr(), ws.data_ptr(),
                                  nbytes, err.data_ptr(), stream)
        assert st == A.OK, A.status_string(st)
        torch.cuda.synchronize()
        outs.append((L.cpu().numpy().copy(), N.cpu().numpy().copy(), idx.cpu().numpy().copy(),
                     int(err.item()) & 0xFFFFFFFF))
    return outs if calls > 1 else outs[0]


def oracle(x, mode, *, gamma=0.5, beta=1.0, select=None):
    sel = slice(None) if select is None else select
    return O.fuse_verify_xvocab(x.logits_full[sel], x.logits_comp[sel], x.logits_ver[sel],
                                x.map_d, x.map_v, x.draft_tokens[sel], x.draft_probs[sel],
                                x.uniforms[sel], dtype=x.dtype, gamma=gamma, beta=beta,
                                mode=mode)


def compare(x, got, o, select=None):
    L, N, I, _ = got
    sel = np.arange(x.B) if select is None else np.asarray(select)
    L, N, I = L[sel], N[sel], I[sel]
    assert np.array_equal(L < 0, o.error) and np.array_equal(N < 0, o.error)
    ok = ~o.flagged & ~o.error
    assert np.array_equal(L[ok], o.accept_len[ok])
    assert np.array_equal(I[ok], o.next_index[ok])
    assert np.array_equal(N[ok], o.next_token[ok])
    # every emitted token is a verifier token of the shared set, its pair's
    good = ~o.error
    assert np.all((I[good] >= 0) & (I[good] < x.S))
    assert np.array_equal(N[good], x.map_v[I[good]])
    return int(ok.sum()), int(o.flagged.sum())


@functools.lru_cache(maxsize=None)
def full_size(cfg, B, K):
    """Cross-family inputs over the paper's shared set (generated once per module)."""
    w = synth.CONFIGS[cfg]
    return synth.make_xvocab(w.recipe, w.seed, B, K, synth.XVOCAB_S, synth.XVOCAB_V_D,
                             synth.XVOCAB_V_V, synth.BF16)


def small(dtype, S, seed=11, B=4, K=3, V_d=300, V_v=250):
    return synth.make_xvocab(synth.CONFIGS[1].recipe, seed, B, K, S, V_d, V_v, dtype)


@pytest.mark.parametrize("mode", [GREEDY, STOCH])
@pytest.mark.parametrize("dtype,S", [(synth.FP32, 200), (synth.BF16, 200), (synth.BF16, 203),
                                     (synth.FP32, 203)])
def test_small_matches_oracle(torch, mode, dtype, S):
    # S * element size a multiple of 16 runs the fast kernel, else the generic one
    x = small(dtype, S)
    compared, flagged = compare(x, run(torch, x, mode), oracle(x, mode))
    assert compared + flagged == x.B


@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_qwen_llama_sized_rows_match_oracle(torch, mode):
    # a Qwen3-sized drafter vocabulary, a Llama-3-sized verifier vocabulary
    # and the paper's shared set (plus two special pairs), config 1's recipe
    x = full_size(1, 8, 5)
    compared, flagged = compare(x, run(torch, x, mode), oracle(x, mode))
    assert compared >= 6


@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_full_batch_sampled_elements(torch, mode):
    # the launch the bench times (B = 64, K = 7, config 2's Zipf recipe over
    # the shared set), compared with the oracle on four batch elements
    x = full_size(2, 64, 7)
    got = run(torch, x, mode)
    sel = np.array([0, 21, 42, 63])
    compared, flagged = compare(x, got, oracle(x, mode, select=sel), select=sel)
    assert compared >= 3
    assert np.all(got[0] >= 0) and got[3] == 0


def test_identity_map_is_the_plain_step(torch):
    # one shared vocabulary, every token paired with itself: the same outputs
    # as asymspec_fuse_verify_ex on the unrestricted rows
    w = synth.CONFIGS[0]
    b = synth.generate(w.recipe, w.seed, 3, 4, 4096, synth.FP32)
    ident = np.arange(4096, dtype=np.int32)
    x = synth.XBatch(b.logits_full, b.logits_comp, b.logits_ver, ident, ident, b.draft_tokens,
                     b.draft_probs, b.uniforms, 3, 4, 4096, 4096, 4096, synth.FP32)
    for mode in (GREEDY, STOCH):
        L, N, I, err = run(torch, x, mode)
        fv = A.FuseVerify(3, 4)
        r = fv(dev(torch, b.logits_full), dev(torch, b.logits_comp), dev(torch, b.logits_ver),
               dev(torch, b.draft_tokens.astype(np.int32)), dev(torch, b.draft_probs),
               dev(torch, b.uniforms), mode=mode)
        torch.cuda.synchronize()
        assert np.array_equal(L, r["accept_len"].cpu().numpy())
        assert np.array_equal(N, r["next_token"].cpu().numpy())
        assert np.array_equal(I, N) and err == 0


def gather(torch, x, md, mv, with_scratch):
    """asymspec_xvocab_gather on a synth.XBatch; the three restricted arrays as
    bit patterns and the error word."""
    rows = x.B * (x.K + 1)
    a, b = dev(torch, x.logits_full, x.dtype), dev(torch, x.logits_comp, x.dtype)
    t = dev(torch, x.logits_ver, x.dtype)
    mdd, mvd = dev(torch, np.asarray(md, np.int32)), dev(torch, np.asarray(mv, np.int32))
    tdt = torch.float32 if x.dtype == synth.FP32 else torch.bfloat16
    outs = [torch.empty(rows, x.S, dtype=tdt, device="cuda") for _ in range(3)]
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    n = A.xvocab_gather_scratch_bytes(x.V_d, x.V_v)
    scratch = torch.full((n,), 0x5A, dtype=torch.uint8, device="cuda") if with_scratch else None
    st = A.xvocab_gather(a.data_ptr(), b.data_ptr(), x.V_d, t.data_ptr(), x.V_v, mdd.data_ptr(),
                         mvd.data_ptr(), x.S, rows, x.dtype, *[o.data_ptr() for o in outs],
                         err.data_ptr(), scratch.data_ptr() if with_scratch else None,
                         n if with_scratch else 0, torch.cuda.current_stream().cuda_stream)
    assert st == A.OK
    torch.cuda.synchronize()
    bits = np.uint32 if x.dtype == synth.FP32 else np.uint16
    got = [o.view(torch.int32 if x.dtype == synth.FP32 else torch.int16).cpu().numpy().view(bits)
           for o in outs]
    return got, int(err.item()) & 0xFFFFFFFF


@pytest.mark.parametrize("with_scratch", [True, False])
@pytest.mark.parametrize("S", [200, 203])
@pytest.mark.parametrize("dtype", [synth.FP32, synth.BF16])
def test_gather_is_exact(torch, dtype, S, with_scratch):
    # with and without the map check, 16-byte and unaligned restricted rows
    x = small(dtype, S, seed=5, B=3, K=2, V_d=1000, V_v=776)
    rows = x.B * (x.K + 1)
    got, err = gather(torch, x, x.map_d, x.map_v, with_scratch)
    bits = np.uint32 if dtype == synth.FP32 else np.uint16
    want = [x.logits_full.reshape(rows, -1)[:, x.map_d], x.logits_comp.reshape(rows, -1)[:, x.map_d],
            x.logits_ver.reshape(rows, -1)[:, x.map_v]]
    for g, w_ in zip(got, want):
        assert np.array_equal(g, w_.view(bits))
    assert err == 0


def test_gather_of_full_size_rows(torch):
    # Qwen3 / Llama-3 sized rows and the paper's shared set
    x = full_size(1, 8, 5)
    rows = x.B * (x.K + 1)
    got, err = gather(torch, x, x.map_d, x.map_v, True)
    assert np.array_equal(got[0], x.logits_full.reshape(rows, -1)[:, x.map_d])
    assert np.array_equal(got[1], x.logits_comp.reshape(rows, -1)[:, x.map_d])
    assert np.array_equal(got[2], x.logits_ver.reshape(rows, -1)[:, x.map_v])
    assert err == 0


@pytest.mark.parametrize("side", ["d", "v"])
def test_a_token_in_two_pairs_is_a_data_error(torch, side):
    # the map check finds the token claimed twice: the map bit is set and
    # every batch element is a data error (pair index included); the gather
    # itself still copies what the maps name
    x = small(synth.BF16, 200, V_d=304, V_v=256)
    md, mv = x.map_d.copy(), x.map_v.copy()
    if side == "d":
        md[40] = md[41]
    else:
        mv[7] = mv[150]
    with pytest.raises(ValueError):
        O.check_vocab_map(md, mv, x.V_d, x.V_v)
    got, err = gather(torch, x, md, mv, True)
    assert err & A.DATA_BAD_MAP
    rows = x.B * (x.K + 1)
    assert np.array_equal(got[0], x.logits_full.reshape(rows, -1)[:, md])
    assert np.array_equal(got[2], x.logits_ver.reshape(rows, -1)[:, mv])
    _, err = gather(torch, x, md, mv, False)           # without the check: not detected
    assert err == 0
    for mode in (GREEDY, STOCH):
        L, N, I, e = run(torch, x, mode, map_d=md, map_v=mv)
        assert np.all(L == -1) and np.all(N == -1) and np.all(I == -1) and e & A.DATA_BAD_MAP


@pytest.mark.parametrize("side", ["d", "v"])
def test_map_entry_outside_its_vocabulary_is_a_data_error(torch, side):
    # never dereferenced: every batch element reports a data error and the
    # map bit is set (the oracle rejects such a map outright)
    x = small(synth.BF16, 200)
    md, mv = x.map_d.copy(), x.map_v.copy()
    if side == "d":
        md[17] = x.V_d
    else:
        mv[150] = -3
    with pytest.raises(ValueError):
        O.check_vocab_map(md, mv, x.V_d, x.V_v)
    for mode in (GREEDY, STOCH):
        L, N, I, err = run(torch, x, mode, map_d=md, map_v=mv)
        assert np.all(L == -1) and np.all(N == -1)
        assert err & A.DATA_BAD_MAP and err & A.DATA_NONFINITE


def test_pair_index_outside_the_shared_set_and_repeat_calls(torch):
    # a draft pair index >= S is that element's data error (as in the oracle);
    # two calls in a row on one workspace give the same results
    x = small(synth.FP32, 200)
    d = x.draft_tokens.copy()
    d[2, 1] = x.S
    x2 = synth.XBatch(**{**x.__dict__, "draft_tokens": d})
    o = oracle(x2, STOCH)
    assert list(o.error) == [False, False, True, False]
    first, second = run(torch, x2, STOCH, calls=2)
    compare(x2, first, o)
    for u, v in zip(first[:3], second[:3]):
        assert np.array_equal(u, v)
    assert first[3] & A.DATA_BAD_TOKEN
