"""The C-ABI library builds, loads and exports what include/asymspec.h declares.

No compute call is made here: only entry points that return before touching
the GPU (argument validation, sizes, strings) are exercised.
"""
import ctypes
import os
import re

import pytest

from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build_cuda()
    return A.lib()


def declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(asymspec_\w+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert names == set(A.EXPORTED)
    for n in names:
        assert hasattr(lib, n), n


def test_library_is_built_for_sm_103a_only(lib):
    # the build command pins one -gencode; this checks the recorded command line
    assert build.GENCODE == "arch=compute_103a,code=sm_103a"


def test_defaults_and_strings(lib):
    g = A.default_gate_params()
    assert (g.gamma, g.beta, g.mode, g.divergence, g.fuse_bonus, g.flags) == (0.5, 1.0, 0, 0, 0, 0)
    assert g.lambda_ == pytest.approx(0.1)
    assert A.status_string(A.OK) == "ok"
    assert "workspace" in A.status_string(A.ERR_WORKSPACE)
    assert A.version() == 200


def _up(n):
    return (n + 255) // 256 * 256


def tma_bytes(B, K, C):
    """Records and tickets, then the cluster kernels' per-row results: a
    48-byte row record of pass 1, and per CTA room for eight 32-byte pass-2
    records (one per warp of the production row kernel) and 80 group masses."""
    R = B * (K + 1)
    return _up(R * 16) + _up(B * 4) + _up(R * 48) + _up(R * C * 8 * 32) + _up(R * C * 80 * 4)


def test_workspace_size():
    # the TMA kernel's layout for clusters of up to 16 CTAs, independent of V
    assert A.workspace_bytes(64, 7, 128256) == tma_bytes(64, 7, 16)
    assert A.workspace_bytes(3, 2, 10) == A.workspace_bytes(3, 2, 10**5) == tma_bytes(3, 2, 16)
    assert A.workspace_bytes(3, 2, 250000) == tma_bytes(3, 2, 16)
    assert A.workspace_bytes(0, 7, 10) == 0
    assert A.workspace_bytes(64, 7, 128256) < 8 << 20


FAKE = 0x10000  # never dereferenced: every call below fails validation first


def call(B=2, K=2, V=64, dtype=A.FP32, gate=None, ws=FAKE, ws_bytes=1 << 20, **ptrs):
    p = dict(a=FAKE, b=FAKE, t=FAKE, tok=FAKE, prob=FAKE, unif=FAKE, L=FAKE, N=FAKE)
    p.update(ptrs)
    return A.fuse_verify_ex(p["a"], p["b"], p["t"], p["tok"], p["prob"], p["unif"], B, K, V,
                            dtype, gate, p["L"], p["N"], ws, ws_bytes)


def test_host_validation_codes(lib):
    assert call(B=0) == A.ERR_INVALID_ARG
    assert call(K=0) == A.ERR_INVALID_ARG
    assert call(V=1) == A.ERR_INVALID_ARG
    assert call(dtype=7) == A.ERR_UNSUPPORTED
    assert call(gate=A.gate_params(gamma=0.0)) == A.ERR_INVALID_ARG
    assert call(gate=A.gate_params(gamma=1.5)) == A.ERR_INVALID_ARG
    assert call(gate=A.gate_params(beta=-1.0)) == A.ERR_INVALID_ARG
    assert call(gate=A.gate_params(beta=float("nan"))) == A.ERR_INVALID_ARG
    assert call(gate=A.gate_params(mode=5)) == A.ERR_UNSUPPORTED
    assert call(gate=A.gate_params(divergence=9)) == A.ERR_UNSUPPORTED
    assert call(a=0) == A.ERR_INVALID_ARG
    assert call(L=0) == A.ERR_INVALID_ARG
    assert call(gate=A.gate_params(mode=A.MODE_STOCHASTIC), prob=0) == A.ERR_INVALID_ARG
    assert call(a=FAKE + 2) == A.ERR_MISALIGNED
    assert call(dtype=A.BF16, a=FAKE + 1) == A.ERR_MISALIGNED
    assert call(tok=FAKE + 2) == A.ERR_MISALIGNED
    assert call(ws=0) == A.ERR_WORKSPACE
    # below even the cluster kernels' records and tickets (2 x 3 rows, 2 tickets)
    assert call(ws_bytes=511) == A.ERR_WORKSPACE
    g = A.GateParams(0.5, 1.0, 0.1, 0, 0, 0, 3)
    assert call(gate=g) == A.ERR_INVALID_ARG          # delta source 3 does not exist
    g = A.GateParams(0.5, 1.0, 0.1, 0, 0, 0, 4)
    assert call(gate=g) == A.ERR_INVALID_ARG          # reserved flag bits must be 0
    opts = A.LaunchOpts(17, 0, 0)
    st = A.fuse_verify_ex(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 2, 64, A.FP32, None, FAKE,
                          FAKE, FAKE, 1 << 20, opts=opts)
    assert st == A.ERR_INVALID_ARG                       # at most 16 CTAs per cluster
    st = A.fuse_verify_ex(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 2, 64, A.FP32, None, FAKE,
                          FAKE, FAKE, 1 << 20, opts=A.LaunchOpts(0, 0, 7))
    assert st == A.ERR_INVALID_ARG                       # unknown kernel
    for removed in (3, 4, 5):                            # numbers of no kernel
        st = A.fuse_verify_ex(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 2, 64, A.FP32, None, FAKE,
                              FAKE, FAKE, 1 << 20, opts=A.LaunchOpts(0, 0, removed))
        assert st == A.ERR_INVALID_ARG
    half = A.LaunchOpts(0, 0, 0, 0, FAKE, 0)             # one timing event without the other
    assert A.fuse_verify_ex(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 2, 64, A.FP32, None, FAKE,
                            FAKE, FAKE, 1 << 20, opts=half) == A.ERR_INVALID_ARG
    for bits in (2, 4, -1):                              # reserved test-flag bits set
        assert A.fuse_verify_ex(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 2, 64, A.FP32, None, FAKE,
                                FAKE, FAKE, 1 << 20, opts=A.LaunchOpts(0, 0, 0, bits)) \
            == A.ERR_INVALID_ARG
    small = tma_bytes(2, 2, 4) - 1                       # TMA kernel forced (clusters of 4), short
    st = A.fuse_verify_ex(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 2, 2, 64, A.FP32, None, FAKE,
                          FAKE, FAKE, small, opts=A.LaunchOpts(4, 0, A.KERNEL_TMA))
    assert st == A.ERR_WORKSPACE


def test_host_entry_point_scratch_layout_and_validation(lib):
    # the device copies of the inputs and outputs, then one workspace per chunk of
    # ceil(B / 8) batch elements, each part 256-byte aligned
    for B, K, V, dtype, elt in ((64, 7, 128256, A.BF16, 2), (13, 3, 4099, A.FP32, 4),
                                (1, 1, 2, A.FP32, 4)):
        R = B * (K + 1)
        Bc = -(-B // A.HOST_CHUNKS)
        P = -(-B // Bc)
        want = (3 * _up(R * V * elt) + 2 * _up(B * K * 4) + _up(R * 4) + 2 * _up(B * 4)
                + _up(_up(A.workspace_bytes(Bc, K, V)) * P))
        assert A.host_scratch_bytes(B, K, V, dtype) == want
    assert A.host_scratch_bytes(0, 7, 10, A.BF16) == 0
    assert A.host_scratch_bytes(2, 2, 10, 7) == 0
    # validation before any CUDA call
    args = (FAKE, FAKE, FAKE, FAKE, FAKE, FAKE)
    need = A.host_scratch_bytes(2, 2, 64, A.FP32)
    assert A.fuse_verify_host(*args, 0, 2, 64, A.FP32, None, FAKE, FAKE, FAKE, need) \
        == A.ERR_INVALID_ARG
    assert A.fuse_verify_host(*args, 2, 2, 64, 9, None, FAKE, FAKE, FAKE, need) == A.ERR_UNSUPPORTED
    assert A.fuse_verify_host(*args, 2, 2, 64, A.FP32, None, 0, FAKE, FAKE, need) \
        == A.ERR_INVALID_ARG
    stoch = A.gate_params(mode=A.MODE_STOCHASTIC)
    assert A.fuse_verify_host(FAKE, FAKE, FAKE, FAKE, 0, FAKE, 2, 2, 64, A.FP32, stoch, FAKE,
                              FAKE, FAKE, need) == A.ERR_INVALID_ARG
    assert A.fuse_verify_host(*args, 2, 2, 64, A.FP32, None, FAKE, FAKE, 0, need) \
        == A.ERR_WORKSPACE
    assert A.fuse_verify_host(*args, 2, 2, 64, A.FP32, None, FAKE, FAKE, FAKE + 16, need) \
        == A.ERR_WORKSPACE                               # not 256-byte aligned
    assert A.fuse_verify_host(*args, 2, 2, 64, A.FP32, None, FAKE, FAKE, FAKE, need - 1) \
        == A.ERR_WORKSPACE


def test_static_entry_point_rejects_batches_above_its_scratch(lib):
    # returns before any CUDA call: B*(K+1) above the static scratch's rows
    args = (FAKE, FAKE, FAKE, FAKE, FAKE, FAKE)
    assert A.fuse_verify_static(*args, 1025, 7, 64, A.FP32, None, FAKE, FAKE) \
        == A.ERR_SCRATCH_LIMIT
    assert A.fuse_verify_static(*args, 1, 8192, 64, A.FP32, None, FAKE, FAKE) \
        == A.ERR_SCRATCH_LIMIT
    assert A.fuse_verify_static(*args, 0, 7, 64, A.FP32, None, FAKE, FAKE) == A.ERR_INVALID_ARG
    assert "8192" in A.status_string(A.ERR_SCRATCH_LIMIT)


def test_draft_sample_validation_codes(lib):
    # every case returns before any CUDA call
    G, S = A.MODE_GREEDY, A.MODE_STOCHASTIC
    d = A.draft_sample
    assert d(FAKE, 4, 64, 7, G, 0, FAKE, FAKE) == A.ERR_UNSUPPORTED        # dtype
    assert d(FAKE, 4, 64, A.BF16, 2, FAKE, FAKE, FAKE) == A.ERR_UNSUPPORTED  # mode
    assert d(FAKE, -1, 64, A.BF16, G, 0, FAKE, FAKE) == A.ERR_INVALID_ARG
    assert d(FAKE, 4, 1, A.BF16, G, 0, FAKE, FAKE) == A.ERR_INVALID_ARG     # V < 2
    assert d(FAKE, 4, A.DRAFT_MAX_V + 1, A.FP32, G, 0, FAKE, FAKE) == A.ERR_TOO_LARGE
    assert d(FAKE, (1 << 27) + 1, 64, A.FP32, G, 0, FAKE, FAKE) == A.ERR_TOO_LARGE
    for c in (-1, 3, 5, 16):
        assert d(FAKE, 4, 64, A.FP32, G, 0, FAKE, FAKE, c) == A.ERR_INVALID_ARG
    assert d(0, 0, 64, A.FP32, S, 0, 0, 0) == A.OK                          # no rows: no-op
    assert d(0, 4, 64, A.FP32, G, 0, FAKE, FAKE) == A.ERR_INVALID_ARG
    assert d(FAKE, 4, 64, A.FP32, G, 0, 0, FAKE) == A.ERR_INVALID_ARG
    assert d(FAKE, 4, 64, A.FP32, G, 0, FAKE, 0) == A.ERR_INVALID_ARG
    assert d(FAKE, 4, 64, A.FP32, S, 0, FAKE, FAKE) == A.ERR_INVALID_ARG     # sampling: uniforms
    assert d(FAKE + 2, 4, 64, A.FP32, G, 0, FAKE, FAKE) == A.ERR_MISALIGNED
    assert d(FAKE + 1, 4, 64, A.BF16, G, 0, FAKE, FAKE) == A.ERR_MISALIGNED
    assert d(FAKE, 4, 64, A.FP32, G, 0, FAKE + 2, FAKE) == A.ERR_MISALIGNED
    assert d(FAKE, 4, 64, A.FP32, S, FAKE + 1, FAKE, FAKE) == A.ERR_MISALIGNED


def test_plan_picks_kernels_and_clusters_that_fit_on_chip(lib):
    assert A.plan(64, 7, 128256, A.BF16).kernel == A.KERNEL_TMA      # the automatic choice
    TMA = A.LaunchOpts(0, 0, A.KERNEL_TMA)
    # the cluster kernel on the bench workload: 8 CTAs of 96 KB per row, two per SM
    info = A.plan(64, 7, 128256, A.BF16, opts=TMA)
    assert info.kernel == A.KERNEL_TMA and info.cluster_size == 8
    assert info.slice_elems == 16032 and info.vector_path == 1
    assert info.ctas == 64 * 8 * 8 and info.smem_bytes <= 113 * 1024
    # Qwen3-sized bf16 rows: 8 CTAs of 112.7 KB, still two per SM
    info = A.plan(8, 5, 151936, A.BF16, opts=TMA)
    assert info.kernel == A.KERNEL_TMA and info.cluster_size == 8
    assert info.smem_bytes <= 113 * 1024
    # fp32 rows of 151,936 entries: 16 CTAs of 113 KB, two per SM
    info = A.plan(256, 4, 151936, A.FP32, opts=TMA)
    assert info.kernel == A.KERNEL_TMA and info.cluster_size == 16
    assert info.smem_bytes <= 113 * 1024
    info = A.plan(1, 4, 32000, A.FP32, opts=TMA)
    assert info.kernel == A.KERNEL_TMA and info.cluster_size == 4
    info = A.plan(2, 2, 4099, A.BF16)
    assert info.vector_path == 0 and info.kernel == A.KERNEL_GENERIC
    assert info.launches == 1 and info.row_kernel == 0
    info = A.plan(64, 7, 128256, A.BF16, A.gate_params(mode=A.MODE_STOCHASTIC))
    assert info.launches == 2 and info.row_kernel == 1
    # the production row kernel: clusters of 6 keep ~97 rows of 770 KB in flight
    # (within the L2 budget; clusters of 5 would hold ~117); warp blocks of 334 vectors
    assert info.cluster_size == 6 and info.slice_elems == 21376 and info.ctas == 512 * 6
    # fewer rows than a wave of clusters of 8: clusters of 8
    small = A.plan(8, 5, 151936, A.BF16, A.gate_params(mode=A.MODE_STOCHASTIC))
    assert small.row_kernel == 1 and small.cluster_size == 8
    info = A.plan(64, 7, 128256, A.BF16, A.gate_params(mode=A.MODE_GREEDY))
    assert info.launches == 2 and info.row_kernel == 0
    with pytest.raises(A.AsymSpecError):
        A.plan(1, 1, 2_000_000, A.FP32)
    info = A.plan(2, 2, 100, A.FP32, opts=A.LaunchOpts(16, 0, 0))
    assert info.cluster_size == 16
    info = A.plan(2, 2, 100, A.FP32, opts=A.LaunchOpts(3, 0, 0))
    assert info.cluster_size == 3
    info = A.plan(64, 7, 128256, A.BF16, opts=A.LaunchOpts(0, 0, A.KERNEL_GENERIC))
    assert info.kernel == A.KERNEL_GENERIC and info.cluster_size == 8
    with pytest.raises(A.AsymSpecError):      # unaligned rows cannot use bulk copies
        A.plan(2, 2, 4099, A.BF16, opts=A.LaunchOpts(0, 0, A.KERNEL_TMA))


def test_row_kernel_plans_fit_on_chip_across_shapes(lib):
    # the production row kernel's plan over batch sizes, row widths and dtypes:
    # a cluster size the planner offers, warp blocks the decision kernel's walk
    # can stage (16 steps of 32 vectors), four CTAs an SM, one cluster per row;
    # a batch smaller than a wave of clusters of 8 keeps 8 whenever it fits
    S = A.gate_params(mode=A.MODE_STOCHASTIC)
    for dtype, elt in ((A.BF16, 2), (A.FP32, 4)):
        ve = 16 // elt
        for V in (4096, 32000, 50000, 109568, 128256, 151936, 200000):
            for B, K in ((1, 4), (8, 5), (32, 8), (64, 7), (256, 4)):
                try:
                    info = A.plan(B, K, V, dtype, S)
                except A.AsymSpecError as e:
                    assert e.status == A.ERR_TOO_LARGE
                    continue
                if not info.row_kernel:
                    continue
                C, W = info.cluster_size, info.slice_elems
                assert C in (4, 5, 6, 7, 8, 10, 12, 16), (dtype, V, B, K, C)
                assert C * W >= V and W % ve == 0 and W - (V + C - 1) // C < ve
                assert -(-(W // ve) // 8) <= 16 * 32
                assert 4 * (info.smem_bytes + 1024) <= 228 * 1024
                assert info.ctas == B * (K + 1) * C and info.block_threads == 256
                if B * (K + 1) * 8 < 152 * 4 and (V + 7) // 8 <= 16 * 256 * ve:
                    assert C == 8


def test_missing_library_raises_instead_of_falling_back(monkeypatch, tmp_path):
    monkeypatch.setattr(A, "_lib", None)
    monkeypatch.setattr(A, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError):
        A.workspace_bytes(1, 1, 2)


def test_xvocab_workspace_layout_and_validation(lib):
    # the restricted rows a', b', t' ([B, K+1, S] each), the emitted pair
    # indices, the gather's scratch (inverse maps and the map-error word), then
    # the step's workspace for a vocabulary of S entries
    for B, K, S, V_d, V_v, dtype, elt in ((64, 7, 109568, 151936, 128256, A.BF16, 2),
                                          (3, 2, 37, 50, 41, A.FP32, 4)):
        R = B * (K + 1)
        scratch = _up(V_d * 4) + _up(V_v * 4) + 256
        assert A.xvocab_gather_scratch_bytes(V_d, V_v) == scratch
        want = 3 * _up(R * S * elt) + _up(B * 4) + scratch + A.workspace_bytes(B, K, S)
        assert A.xvocab_workspace_bytes(B, K, S, V_d, V_v, dtype) == want
    assert A.xvocab_workspace_bytes(0, 2, 10, 30, 20, A.FP32) == 0
    assert A.xvocab_workspace_bytes(2, 2, 1, 30, 20, A.FP32) == 0
    assert A.xvocab_workspace_bytes(2, 2, 10, 0, 20, A.FP32) == 0
    assert A.xvocab_workspace_bytes(2, 2, 10, 30, 20, 5) == 0
    assert A.xvocab_gather_scratch_bytes(0, 5) == 0
    need = A.xvocab_workspace_bytes(2, 2, 10, 30, 20, A.FP32)

    def fv(B=2, K=2, S=10, V_d=30, V_v=20, dtype=A.FP32, gate=None, ws=FAKE, n=need, **p):
        x = dict(a=FAKE, b=FAKE, t=FAKE, md=FAKE, mv=FAKE, d=FAKE, pr=FAKE, u=FAKE, L=FAKE,
                 N=FAKE, I=0)
        x.update(p)
        return A.fuse_verify_xvocab(x["a"], x["b"], V_d, x["t"], V_v, x["md"], x["mv"], S,
                                    x["d"], x["pr"], x["u"], B, K, dtype, gate, x["L"], x["N"],
                                    x["I"], ws, n)

    # every case returns before any CUDA call
    assert fv(B=0) == A.ERR_INVALID_ARG
    assert fv(S=1) == A.ERR_INVALID_ARG
    assert fv(V_v=0) == A.ERR_INVALID_ARG
    assert fv(dtype=3) == A.ERR_UNSUPPORTED
    assert fv(gate=A.gate_params(gamma=2.0)) == A.ERR_INVALID_ARG
    assert fv(d=0) == A.ERR_INVALID_ARG
    assert fv(gate=A.gate_params(mode=A.MODE_STOCHASTIC), u=0) == A.ERR_INVALID_ARG
    assert fv(N=FAKE + 2) == A.ERR_MISALIGNED
    assert fv(ws=0) == A.ERR_WORKSPACE
    assert fv(ws=FAKE + 16) == A.ERR_WORKSPACE           # not 256-byte aligned
    assert fv(n=need - 1) == A.ERR_WORKSPACE
    assert fv(md=0) == A.ERR_INVALID_ARG                 # the gather's own checks
    assert fv(a=FAKE + 2) == A.ERR_MISALIGNED
    assert fv(mv=FAKE + 1) == A.ERR_MISALIGNED
    g = A.xvocab_gather
    assert g(FAKE, FAKE, 30, FAKE, 20, FAKE, FAKE, 10, -1, A.FP32, FAKE, FAKE, FAKE) \
        == A.ERR_INVALID_ARG
    assert g(0, 0, 30, 0, 20, 0, 0, 10, 0, A.FP32, 0, 0, 0) == A.OK  # no rows: no-op
    assert g(FAKE, FAKE, 30, FAKE, 20, FAKE, FAKE, 10, 4, 9, FAKE, FAKE, FAKE) \
        == A.ERR_UNSUPPORTED
    assert g(FAKE, FAKE, 30, FAKE, 20, FAKE, FAKE, 10, 4, A.BF16, FAKE + 1, FAKE, FAKE) \
        == A.ERR_MISALIGNED
    assert g(FAKE, FAKE, 30, FAKE, 20, FAKE, FAKE, 10, 8 * 65536, A.FP32, FAKE, FAKE, FAKE) \
        == A.ERR_TOO_LARGE
    small = A.xvocab_gather_scratch_bytes(30, 20) - 1
    assert g(FAKE, FAKE, 30, FAKE, 20, FAKE, FAKE, 10, 4, A.FP32, FAKE, FAKE, FAKE, None,
             FAKE, small) == A.ERR_WORKSPACE
    assert g(FAKE, FAKE, 30, FAKE, 20, FAKE, FAKE, 10, 4, A.FP32, FAKE, FAKE, FAKE, None,
             FAKE + 16, small + 1) == A.ERR_WORKSPACE
