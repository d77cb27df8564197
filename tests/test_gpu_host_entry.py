"""asymspec_fuse_verify_host: the step from host memory, pipelined in chunks.

Its outputs must equal, element for element, those of asymspec_fuse_verify_ex
on the same inputs already in device memory (the same kernels run on each
chunk of batch elements), whether the host buffers are page-locked or
pageable, for chunk counts that do and do not divide the batch; and they
are checked against the oracle.
"""
import numpy as np
import pytest

from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth
from tests._parity import device_inputs, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as _torch
    assert _torch.cuda.is_available(), "the gpu tests need a CUDA device"
    from paper_2608_26004_gb300 import build
    build.build_cuda()
    A.lib()
    return _torch


def host_inputs(batch, torch, pinned):
    def t(x):
        x = np.ascontiguousarray(x)
        if batch.dtype == synth.BF16 and x.dtype == np.uint16:
            x = torch.from_numpy(x.view(np.int16)).view(torch.bfloat16)
        else:
            x = torch.from_numpy(x)
        return x.pin_memory() if pinned else x
    return dict(a=t(batch.logits_full), b=t(batch.logits_comp), t=t(batch.logits_ver),
                tokens=t(np.asarray(batch.draft_tokens, np.int32)),
                probs=t(np.asarray(batch.draft_probs, np.float32)),
                unif=t(np.asarray(batch.uniforms, np.float32)))


def run_host(batch, torch, mode, pinned):
    h = host_inputs(batch, torch, pinned)
    L = torch.full((batch.B,), -7, dtype=torch.int32)
    N = torch.full((batch.B,), -7, dtype=torch.int32)
    if pinned:
        L, N = L.pin_memory(), N.pin_memory()
    nbytes = A.host_scratch_bytes(batch.B, batch.K, batch.V, batch.dtype)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    gate = A.gate_params(mode=mode)
    st = A.fuse_verify_host(h["a"].data_ptr(), h["b"].data_ptr(), h["t"].data_ptr(),
                            h["tokens"].data_ptr(), h["probs"].data_ptr(), h["unif"].data_ptr(),
                            batch.B, batch.K, batch.V, batch.dtype, gate, L.data_ptr(),
                            N.data_ptr(), scratch.data_ptr(), nbytes, stream)
    assert st == A.OK, A.status_string(st)
    torch.cuda.synchronize()
    return L.numpy().copy(), N.numpy().copy()


def run_device(batch, torch, mode):
    x = device_inputs(batch, torch)
    fv = A.FuseVerify(batch.B, batch.K)
    res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=mode)
    torch.cuda.synchronize()
    return res["accept_len"].cpu().numpy(), res["next_token"].cpu().numpy()


CASES = [
    (13, 3, 40000, synth.BF16, 61),   # 7 chunks of 2 batch elements (the last holds 1)
    (64, 7, 8200, synth.BF16, 62),    # 8 chunks of 8
    (5, 2, 4099, synth.FP32, 63),     # unaligned rows: the generic kernel in every chunk
    (1, 4, 32000, synth.FP32, 64),    # one chunk
]


@pytest.mark.parametrize("case", range(len(CASES)))
@pytest.mark.parametrize("mode", [A.MODE_GREEDY, A.MODE_STOCHASTIC])
def test_host_entry_point_matches_the_device_entry_point(torch, case, mode):
    B, K, V, dtype, seed = CASES[case]
    batch = synth.generate(synth.Recipe(), seed, B, K, V, dtype)
    Ld, Nd = run_device(batch, torch, mode)
    for pinned in (True, False):
        Lh, Nh = run_host(batch, torch, mode, pinned)
        assert np.array_equal(Lh, Ld) and np.array_equal(Nh, Nd), f"pinned={pinned}"
    o = run_oracle(batch, mode=mode)
    ok = ~o.flagged & ~o.error
    assert np.array_equal(Ld[ok], o.accept_len[ok]) and np.array_equal(Nd[ok], o.next_token[ok])


def test_host_entry_point_reuses_a_scratch_across_batch_sizes(torch):
    # the chunk tickets are cleared by every call, so one scratch serves any batch it fits
    big = synth.generate(synth.Recipe(), 71, 16, 3, 4099, synth.FP32)
    small = synth.generate(synth.Recipe(), 72, 3, 3, 4099, synth.FP32)
    nbytes = A.host_scratch_bytes(16, 3, 4099, synth.FP32)
    scratch = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    for batch in (big, small, big):
        h = host_inputs(batch, torch, True)
        L = torch.empty(batch.B, dtype=torch.int32).pin_memory()
        N = torch.empty(batch.B, dtype=torch.int32).pin_memory()
        st = A.fuse_verify_host(h["a"].data_ptr(), h["b"].data_ptr(), h["t"].data_ptr(),
                                h["tokens"].data_ptr(), h["probs"].data_ptr(),
                                h["unif"].data_ptr(), batch.B, batch.K, batch.V, batch.dtype,
                                None, L.data_ptr(), N.data_ptr(), scratch.data_ptr(), nbytes,
                                stream)
        assert st == A.OK
        torch.cuda.synchronize()
        Ld, Nd = run_device(batch, torch, A.MODE_GREEDY)
        assert np.array_equal(L.numpy(), Ld) and np.array_equal(N.numpy(), Nd)
