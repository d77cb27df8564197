"""asymspec_fuse_verify_static: the step with its scratch in a static device array.

The file name sorts last so that these calls also run after every other GPU
test has used the library in the same process; the tests must pass both
alone and then.  Every result is compared bit for bit with
asymspec_fuse_verify_ex given a caller-owned zeroed workspace of the static
scratch's size, which selects the same kernel, on the same inputs, over two
consecutive calls, so that the second call sees the scratch the first one
left; and, on a sample of batch elements, with the float64 oracle.
"""
import numpy as np
import pytest

from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth
from tests._parity import check_decisions, device_inputs, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as _torch
    assert _torch.cuda.is_available(), "the gpu tests need a CUDA device"
    from paper_2608_26004_gb300 import build
    build.build_cuda()
    A.lib()
    return _torch


def _ptr(t):
    return int(t.data_ptr())


def run_static(torch, x, B, K, V, dtype, gate):
    L = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    N = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    st = A.fuse_verify_static(_ptr(x["a"]), _ptr(x["b"]), _ptr(x["t"]), _ptr(x["tokens"]),
                              _ptr(x["probs"]), _ptr(x["unif"]), B, K, V, dtype, gate,
                              _ptr(L), _ptr(N), stream)
    assert st == A.OK, A.status_string(st)
    torch.cuda.synchronize()
    return L.cpu().numpy(), N.cpu().numpy()


def run_ex(torch, x, B, K, V, dtype, gate):
    """The workspace entry point with a workspace of the static scratch's size:
    the automatic choice then takes the kernel the static entry takes."""
    L = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    N = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    nbytes = A.STATIC_SCRATCH_BYTES
    ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    st = A.fuse_verify_ex(_ptr(x["a"]), _ptr(x["b"]), _ptr(x["t"]), _ptr(x["tokens"]),
                          _ptr(x["probs"]), _ptr(x["unif"]), B, K, V, dtype, gate, _ptr(L),
                          _ptr(N), _ptr(ws), nbytes, stream=stream)
    assert st == A.OK, A.status_string(st)
    torch.cuda.synchronize()
    return L.cpu().numpy(), N.cpu().numpy()


CASES = [
    # (B, K, V, dtype, mode, seed): the second call reuses the scratch the first left
    (8, 5, 151936, synth.BF16, A.MODE_STOCHASTIC, 11),
    (3, 2, 4099, synth.BF16, A.MODE_GREEDY, 12),          # unaligned rows: generic kernel
    (1024, 7, 64, synth.FP32, A.MODE_STOCHASTIC, 13),     # B*(K+1) = the 8192-row limit
    (1024, 7, 64, synth.FP32, A.MODE_GREEDY, 14),
    (64, 7, 128256, synth.BF16, A.MODE_STOCHASTIC, 15),   # 512 rows: the TMA kernel
    (700, 7, 12288, synth.FP32, A.MODE_GREEDY, 16),       # TMA part too large: generic
]


@pytest.mark.parametrize("first,second", [(0, 1), (2, 3), (3, 0), (4, 5), (5, 4)])
def test_two_consecutive_calls_match_the_workspace_entry_point(torch, first, second):
    for idx in (first, second):
        B, K, V, dtype, mode, seed = CASES[idx]
        batch = synth.generate(synth.Recipe(), seed, B, K, V, dtype)
        x = device_inputs(batch, torch)
        gate = A.gate_params(mode=mode)
        Ls, Ns = run_static(torch, x, B, K, V, dtype, gate)
        Le, Ne = run_ex(torch, x, B, K, V, dtype, gate)
        assert np.array_equal(Ls, Le) and np.array_equal(Ns, Ne), f"case {idx} differs"
        assert np.all(Ls >= 0) and np.all(Ls <= K) and np.all(Ns >= 0) and np.all(Ns < V)
        # a sample of the elements against the oracle: first, last, and six more
        rng = np.random.default_rng(seed)
        sel = np.unique(np.concatenate([[0, B - 1], rng.choice(B, size=min(B, 6), replace=False)]))
        o = run_oracle(batch, mode=mode, select=sel, logprobs=False)
        check_decisions(batch, sel, Ls[sel], Ns[sel], o, mode)


def test_rows_above_the_limit_are_rejected_before_any_launch(torch):
    B, K, V = 1025, 7, 64                                 # 8200 rows > 8192
    x = dict(a=torch.zeros(B * (K + 1) * V, device="cuda"))
    L = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    st = A.fuse_verify_static(_ptr(x["a"]), _ptr(x["a"]), _ptr(x["a"]), _ptr(L), 0, 0, B, K,
                              V, synth.FP32, None, _ptr(L), _ptr(L), 0)
    assert st == A.ERR_SCRATCH_LIMIT
    assert "8192" in A.status_string(st)
    torch.cuda.synchronize()
    assert np.all(L.cpu().numpy() == -7)                  # nothing ran


def _up(n):
    return (n + 255) // 256 * 256


def test_the_cases_cover_both_kernels_the_scratch_selects(torch):
    # the cluster kernels need, beyond records and tickets, 48 bytes per row
    # and 576 per row and CTA; the static scratch takes them when these fit
    fits = []
    for B, K, V, dtype, mode, seed in CASES:
        info = A.plan(B, K, V, dtype, A.gate_params(mode=mode))
        R = B * (K + 1)
        need = (_up(R * 16) + _up(B * 4) + _up(R * 48) + _up(R * info.cluster_size * 256)
                + _up(R * info.cluster_size * 320))
        if info.kernel == A.KERNEL_TMA:
            fits.append(need <= A.STATIC_SCRATCH_BYTES)
    assert True in fits and False in fits
