"""The persistent form of the cluster kernel (ASYMSPEC_KERNEL_PERSIST).

As many clusters as the device holds each take every G-th row, and each
CTA refills its slice with the cluster's next row chunk by chunk as pass 2
finishes with it.  The per-row arithmetic is the one-shot kernel's, so on the
same inputs the two must agree exactly on every batch element; both are
compared with the oracle as well (bit-exact except the near-ties it flags).
Only the production program sets exist in this form (no debug outputs), so
the outputs compared are the accepted length and the next token.
"""
import numpy as np
import pytest

from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth
from tests._parity import device_inputs, run_oracle

pytestmark = pytest.mark.gpu

GREEDY, STOCH = A.MODE_GREEDY, A.MODE_STOCHASTIC
TMA, PERSIST = A.KERNEL_TMA, A.KERNEL_PERSIST


@pytest.fixture(scope="module")
def torch():
    import torch as _torch
    assert _torch.cuda.is_available(), "the gpu tests need a CUDA device"
    from paper_2608_26004_gb300 import build
    build.build_cuda()
    A.lib()
    return _torch


def run(batch, torch, x, kernel, **kw):
    fv = A.FuseVerify(batch.B, batch.K)
    res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], kernel=kernel, **kw)
    torch.cuda.synchronize()
    return res["accept_len"].cpu().numpy(), res["next_token"].cpu().numpy()


def against_oracle(batch, L, N, select=None, **kw):
    o = run_oracle(batch, select=select, logprobs=False, **kw)
    sel = np.arange(batch.B) if select is None else np.asarray(select)
    L, N = L[sel], N[sel]
    ok = ~o.flagged & ~o.error
    assert np.array_equal(L < 0, o.error) and np.array_equal(N < 0, o.error)
    assert np.array_equal(L[ok], o.accept_len[ok]) and np.array_equal(N[ok], o.next_token[ok])
    return int(ok.sum())


def both_kernels(batch, torch, **kw):
    x = device_inputs(batch, torch)
    L1, N1 = run(batch, torch, x, TMA, **kw)
    L2, N2 = run(batch, torch, x, PERSIST, **kw)
    assert np.array_equal(L1, L2) and np.array_equal(N1, N2), "persistent != one-shot"
    return L2, N2


SMALL = [(6, 3, 40000, synth.BF16, 41), (4, 2, 8200, synth.FP32, 42), (5, 2, 8, synth.BF16, 43),
         (3, 3, 1000, synth.FP32, 44), (7, 4, 16384 * 3 + 8, synth.BF16, 45)]


@pytest.mark.parametrize("div", [A.DIV_JSD, A.DIV_KL, A.DIV_NONE, A.DIV_LAMBDA])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_small_batches(torch, div, mode):
    for B, K, V, dtype, seed in SMALL:
        batch = synth.generate(synth.Recipe(), seed, B, K, V, dtype)
        for fuse_bonus in ((False, True) if mode == GREEDY else (False,)):
            kw = dict(mode=mode, divergence=div, fuse_bonus=fuse_bonus)
            L, N = both_kernels(batch, torch, **kw)
            assert against_oracle(batch, L, N, **kw) > 0


@pytest.mark.parametrize("cfg,nb", [(1, None), (2, None), (3, 40), (4, 12)])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_workloads(torch, cfg, nb, mode):
    # every cluster takes several rows (512 rows at B = 64, K = 7); all batch
    # elements against the one-shot kernel, four against the oracle
    batch = synth.make_config(cfg, sweep_index=3 if cfg == 4 else 0, nb=nb)
    L, N = both_kernels(batch, torch, mode=mode)
    sel = np.array([0, batch.B // 3, (2 * batch.B) // 3, batch.B - 1])
    assert against_oracle(batch, L, N, select=sel, mode=mode) >= 2


@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_entries_far_above_the_first_vector(torch, mode):
    # the fixed-reference sums overflow and a CTA redoes its slice with a
    # running maximum, in a row that is not the cluster's first
    batch = synth.generate(synth.Recipe(), 91, 40, 2, 40000, synth.BF16)
    bits = np.zeros(1, np.float32)
    bits[0] = 150.0
    spike = (bits.view(np.uint32) >> 16).astype(np.uint16)[0]
    for arr in (batch.logits_full, batch.logits_comp, batch.logits_ver):
        arr[0, 1, 30001] = spike
        arr[39, 2, 12345] = spike
    L, N = both_kernels(batch, torch, mode=mode)
    assert against_oracle(batch, L, N, mode=mode) > 30


def test_debug_outputs_are_not_offered(torch):
    batch = synth.generate(synth.Recipe(), 7, 2, 2, 8200, synth.BF16)
    x = device_inputs(batch, torch)
    fv = A.FuseVerify(batch.B, batch.K)
    with pytest.raises(A.AsymSpecError) as e:
        fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=STOCH,
           row_stats=True, kernel=PERSIST)
    assert e.value.status == A.ERR_UNSUPPORTED
    info = A.plan(64, 7, 128256, A.BF16, A.gate_params(mode=STOCH),
                  A.LaunchOpts(0, 0, PERSIST))
    assert info.kernel == PERSIST and info.cluster_size == 8
    assert info.ctas == info.max_active_clusters * 8 and 0 < info.ctas <= 512 * 8
