"""GPU path (through the C ABI) against the float64 oracle on the same inputs.

Every case runs on the kernel the library picks (for 16-byte aligned rows
the one-shot cluster kernels, the generic kernel otherwise) and on the
generic kernel: with accepted lengths and next tokens only (the production
program the benchmark times: in stochastic mode with the JSD gate, the
production row kernel), with the per-row tokens as well, and with every
debug output (row statistics, fused log-probs), which runs the full per-row
program.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_26004_gb300 import asymspec as A
from paper_2608_26004_gb300 import synth
from tests._parity import check_decisions, compare, device_inputs, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

GREEDY, STOCH = A.MODE_GREEDY, A.MODE_STOCHASTIC
AUTO, GENERIC, TMA = A.KERNEL_AUTO, A.KERNEL_GENERIC, A.KERNEL_TMA
# the automatic choice (the one-shot cluster kernels for aligned rows) and
# the generic cluster kernel; "row": outputs of the production program only
PATHS = [(AUTO, "row"), (AUTO, False), (AUTO, True), (GENERIC, True)]
PATH_IDS = ["auto-row", "auto-prod", "auto-full", "generic-full"]


@pytest.fixture(scope="module")
def torch():
    import torch as _torch
    assert _torch.cuda.is_available(), "the gpu tests need a CUDA device"
    from paper_2608_26004_gb300 import build
    build.build_cuda()
    A.lib()
    return _torch


def small(B, K, V, dtype, seed, **kw):
    rc = synth.Recipe(**kw) if kw else synth.Recipe()
    return synth.generate(rc, seed, B, K, V, dtype)


def check(batch, torch, mode, kernel, full, **kw):
    g = run_gpu(batch, torch, mode=mode, kernel=kernel, full=full, **kw)
    okw = {k: v for k, v in kw.items()
           if k in ("divergence", "gamma", "beta", "lam", "fuse_bonus", "delta_source")}
    o = run_oracle(batch, mode=mode, **okw)
    compare(batch, g, o, mode=mode)
    return g, o


# ---------------------------------------------------------------- element by element

SMALL = [
    # B, K, V, dtype          (TMA kernel iff V * element size % 16 == 0)
    (3, 3, 1000, synth.FP32),     # 250 float4 per row
    (2, 2, 4099, synth.BF16),     # odd V: generic kernel, scalar path, ragged tail
    (4, 1, 8200, synth.BF16),     # 1025 uint4 per row
    (2, 4, 33333, synth.FP32),    # generic kernel, scalar path, multi-CTA clusters
    (5, 2, 2, synth.FP32),        # smallest vocabulary
    (2, 2, 8, synth.BF16),        # one 16-byte vector per row
    (3, 2, 40000, synth.BF16),    # several rounds and bulk-copy chunks per CTA
]


@pytest.mark.parametrize("kernel,full", PATHS, ids=PATH_IDS)
@pytest.mark.parametrize("B,K,V,dtype", SMALL)
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_small_shapes(torch, B, K, V, dtype, mode, kernel, full):
    batch = small(B, K, V, dtype, seed=1000 + V + K)
    check(batch, torch, mode, kernel, full)


@pytest.mark.parametrize("kernel", [GENERIC, TMA])
@pytest.mark.parametrize("cluster", [1, 2, 3, 4, 8, 16])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_forced_cluster_sizes(torch, cluster, mode, kernel):
    for B, K, V, dtype in [(3, 2, 5000, synth.BF16), (2, 2, 780, synth.FP32),
                           (2, 1, 16, synth.BF16)]:
        batch = small(B, K, V, dtype, seed=77 + cluster + V)
        for full in (False, True):
            check(batch, torch, mode, kernel, full, cluster_size=cluster)


@pytest.mark.parametrize("kernel,full", PATHS, ids=PATH_IDS)
@pytest.mark.parametrize("div", [A.DIV_JSD, A.DIV_NONE, A.DIV_KL, A.DIV_LAMBDA])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_gate_variants(torch, div, mode, kernel, full):
    batch = small(4, 3, 6000, synth.BF16, seed=300 + div, sigma_c=2.0, frac_lo=0.1, frac_hi=0.3)
    check(batch, torch, mode, kernel, full, divergence=div, lam=0.1)


@pytest.mark.parametrize("kernel,full", PATHS, ids=PATH_IDS)
@pytest.mark.parametrize("gamma,beta,fuse_bonus", [(1.0, 0.0, False), (0.3, 2.0, True),
                                                   (0.7, 0.5, False), (1.0, 1.0, True)])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_hyperparameters(torch, gamma, beta, fuse_bonus, mode, kernel, full):
    batch = small(4, 3, 3000, synth.FP32, seed=int(gamma * 10 + beta * 100))
    check(batch, torch, mode, kernel, full, gamma=gamma, beta=beta, fuse_bonus=fuse_bonus)


# ---------------------------------------------------------------- the five workloads

@pytest.mark.parametrize("kernel,full", PATHS, ids=PATH_IDS)
@pytest.mark.parametrize("cfg", [0, 1])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_small_workloads_whole(torch, cfg, mode, kernel, full):
    batch = synth.make_config(cfg)
    check(batch, torch, mode, kernel, full)


def _bench_call(batch, torch, x, mode):
    """The call bench.py times: no debug outputs, automatic launch."""
    fv = A.FuseVerify(batch.B, batch.K)
    res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=mode)
    torch.cuda.synchronize()
    return res["accept_len"].cpu().numpy(), res["next_token"].cpu().numpy()


@pytest.mark.parametrize("cfg", [2, 3])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_large_workloads_sampled(torch, cfg, mode):
    batch = synth.make_config(cfg)
    x = device_inputs(batch, torch)
    L, N = _bench_call(batch, torch, x, mode)
    rng = np.random.default_rng(cfg * 10 + mode)
    sel = np.sort(rng.choice(batch.B, size=8, replace=False))
    if cfg == 3:  # both halves: z_c == z_f and high divergence
        sel = np.unique(np.concatenate([sel, [0, batch.B // 2 - 1, batch.B // 2, batch.B - 1]]))
    o = run_oracle(batch, mode=mode, select=sel, logprobs=True)
    check_decisions(batch, sel, L[sel], N[sel], o, mode)
    for full in (False, True):
        g = run_gpu(batch, torch, mode=mode, inputs=x, full=full)
        # the production kernel and the full-program kernel sum in different
        # orders: they may differ only on elements where both are correct
        # emissions, checked against the oracle (near-ties of a few 1e-7)
        diff = np.nonzero((g["accept_len"] != L) | (g["next_token"] != N))[0]
        assert diff.size <= 2, f"{diff.size} elements differ between the kernels"
        if diff.size:
            od = run_oracle(batch, mode=mode, select=diff, logprobs=False)
            check_decisions(batch, diff, L[diff], N[diff], od, mode)
            check_decisions(batch, diff, g["accept_len"][diff], g["next_token"][diff], od, mode)
        compare(batch, g, o, mode=mode, select=sel)


@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_divergence_sweep_gate_response(torch, mode):
    rows = []
    flagged = total = 0
    for si, s in enumerate(synth.CONFIGS[4].sweep):
        batch = synth.make_config(4, sweep_index=si)
        o = run_oracle(batch, mode=mode, logprobs=False)
        gp = run_gpu(batch, torch, mode=mode, full=False)
        c = compare(batch, gp, o, mode=mode, logprobs=False, max_flagged=0.125)
        flagged += c["flagged"]
        total += batch.B
        g = run_gpu(batch, torch, mode=mode, logprobs=False)
        compare(batch, g, o, mode=mode, logprobs=False)
        hist_g = np.bincount(gp["accept_len"], minlength=batch.K + 1)
        hist_o = np.bincount(o.accept_len, minlength=batch.K + 1)
        nflag = int(o.flagged.sum())
        assert np.abs(hist_g - hist_o).sum() <= 2 * nflag
        rows.append((s, float(np.mean(g["row_stats"][:, :batch.K, 4])),
                     float(np.mean(g["row_stats"][:, :batch.K, 5]))))
    # near-ties over the six points (the oracle flags 9 of 192 stochastic
    # elements and none of the greedy ones; each is checked for validity)
    assert flagged <= 0.06 * total, f"{flagged} of {total} elements flagged"
    # the gate relaxes as the compressed context diverges: mean D rises,
    # mean gamma_eff falls, from D = 0 at s = 0 (z_c == z_f)
    Ds = [r[1] for r in rows]
    gs = [r[2] for r in rows]
    assert Ds[0] == pytest.approx(0.0, abs=1e-5)
    assert all(np.diff(Ds) > 0) and all(np.diff(gs) < 0)


# ---------------------------------------------------------------- edge cases

@pytest.mark.parametrize("kernel,full", PATHS, ids=PATH_IDS)
def test_data_errors_never_trap(torch, kernel, full):
    batch = small(7, 2, 1000, synth.FP32, seed=5)
    batch.logits_full[1, 0, 17] = np.nan
    batch.logits_ver[2, 2, 999] = np.inf
    batch.draft_tokens[3, 1] = 1000
    batch.draft_tokens[4, 0] = -3
    batch.logits_comp[6, 2, 5] = np.nan      # bonus row: unused by greedy decoding
    for mode in (GREEDY, STOCH):
        g = run_gpu(batch, torch, mode=mode, kernel=kernel, full=full)
        o = run_oracle(batch, mode=mode)
        compare(batch, g, o, mode=mode, check_stats=False, logprobs=False)
        assert list(g["accept_len"][1:5]) == [-1] * 4 and list(g["next_token"][1:5]) == [-1] * 4
        assert g["accept_len"][0] >= 0 and g["accept_len"][5] >= 0
        assert (g["accept_len"][6] >= 0) == (mode == GREEDY)
        word = int(g["error_word"][0])
        assert word & A.DATA_NONFINITE and word & A.DATA_BAD_TOKEN
        assert not word & A.DATA_TIMEOUT
    batch = small(3, 2, 1000, synth.FP32, seed=6)
    batch.draft_probs[0, 1] = 0.0
    batch.uniforms[1, 2] = 1.0
    g = run_gpu(batch, torch, mode=STOCH, kernel=kernel, full=full)
    assert list(g["accept_len"])[:2] == [-1, -1] and g["accept_len"][2] >= 0
    word = int(g["error_word"][0])
    assert word & A.DATA_BAD_PROB and word & A.DATA_BAD_UNIFORM


@pytest.mark.parametrize("delta", [A.DELTA_A, A.DELTA_TB])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
@pytest.mark.parametrize("kernel,full", [(AUTO, False), (AUTO, True), (GENERIC, True)],
                         ids=["auto-prod", "auto-full", "generic-full"])
def test_delta_sources(torch, delta, mode, kernel, full):
    # the mechanism ablation's alternatives to a - b (raw-augmented a, SCD-style
    # t - b): every row quantity and decision against the oracle, aligned and
    # unaligned rows, greedy with and without the fused bonus
    for B, K, V, dtype, seed in ((3, 3, 40000, synth.BF16, 91), (2, 2, 4099, synth.FP32, 92)):
        batch = small(B, K, V, dtype, seed)
        for fuse_bonus in ((False, True) if mode == GREEDY else (False,)):
            check(batch, torch, mode, kernel, full, delta_source=delta, fuse_bonus=fuse_bonus)


@pytest.mark.parametrize("div", [A.DIV_JSD, A.DIV_KL, A.DIV_NONE, A.DIV_LAMBDA])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
@pytest.mark.parametrize("kernel", [AUTO, GENERIC])
def test_accept_and_next_only(torch, div, mode, kernel):
    # no per-row outputs: the program sets the benchmark runs (one production
    # configuration per kernel); accepted length and next token against the
    # oracle, bit-exact except near-ties the oracle flags
    for B, K, V, dtype, seed in ((6, 3, 40000, synth.BF16, 41), (4, 2, 8200, synth.FP32, 42)):
        batch = small(B, K, V, dtype, seed)
        for fuse_bonus in ((False, True) if mode == GREEDY else (False,)):
            x = device_inputs(batch, torch)
            fv = A.FuseVerify(batch.B, batch.K)
            res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=mode,
                     divergence=div, fuse_bonus=fuse_bonus, kernel=kernel)
            torch.cuda.synchronize()
            L, N = res["accept_len"].cpu().numpy(), res["next_token"].cpu().numpy()
            o = run_oracle(batch, mode=mode, divergence=div, fuse_bonus=fuse_bonus)
            assert np.array_equal(L < 0, o.error) and np.array_equal(N < 0, o.error)
            check_decisions(batch, np.arange(batch.B), L, N, o, mode)
            assert (~o.flagged & ~o.error).any()


@pytest.mark.parametrize("kernel", [GENERIC, TMA])
def test_exact_ties_resolve_to_lowest_index(torch, kernel):
    B, K, V = 2, 2, 4096
    a = np.zeros((B, K + 1, V), np.float32)
    b = np.zeros_like(a)
    t = np.zeros_like(a)
    t[..., [100, 3000, 4095]] = 5.0      # three-way tie in t and in s
    t[1, :, [5, 4000]] = 7.0
    batch = synth.Batch(a, b, t, np.full((B, K), 7, np.int32), np.full((B, K), 0.5, np.float32),
                        np.full((B, K + 1), 0.5, np.float32), B, K, V, synth.FP32)
    for cluster in (0, 1, 4, 16):
        for full in (False, True):
            g = run_gpu(batch, torch, mode=GREEDY, cluster_size=cluster, gamma=1.0,
                        kernel=kernel, full=full, fuse_bonus=True)
            assert list(g["row_tokens"][0, :, 0]) == [100] * (K + 1)
            assert list(g["row_tokens"][1, :, 0]) == [5] * (K + 1)
            g = run_gpu(batch, torch, mode=GREEDY, cluster_size=cluster, gamma=1.0,
                        kernel=kernel, full=full)
            assert g["row_tokens"][0, K, 1] == 100 and g["row_tokens"][1, K, 1] == 5


def test_identical_contexts_give_zero_divergence(torch):
    batch = synth.make_config(3, b0=120, nb=4)          # b < 128: z_c == z_f
    g = run_gpu(batch, torch, mode=GREEDY)
    assert np.all(np.abs(g["row_stats"][:2, :, 4]) <= 1e-5)
    assert np.all(np.abs(g["row_stats"][:2, :, 5] - 0.5) <= 1e-5)


def test_misaligned_rows_take_the_generic_kernel(torch):
    batch = small(2, 2, 2048, synth.BF16, seed=9)
    x = device_inputs(batch, torch)
    for key in ("a", "b", "t"):
        buf = torch.empty(x[key].numel() + 1, dtype=x[key].dtype, device="cuda")
        buf[1:].copy_(x[key].reshape(-1))
        x[key] = buf[1:].view(x[key].shape)          # 2-byte aligned, not 16
    assert x["a"].data_ptr() % 16 != 0
    for full in (False, True):
        g = run_gpu(batch, torch, mode=STOCH, inputs=x, full=full)
        o = run_oracle(batch, mode=STOCH)
        compare(batch, g, o, mode=STOCH)


def test_workspace_reuse_and_allocating_entry_point(torch):
    batch = synth.make_config(1)
    x = device_inputs(batch, torch)
    fv = A.FuseVerify(batch.B, batch.K)
    outs = []
    for _ in range(3):
        r = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=STOCH)
        outs.append((r["accept_len"].clone(), r["next_token"].clone()))
    torch.cuda.synchronize()
    for L, N in outs[1:]:
        assert torch.equal(L, outs[0][0]) and torch.equal(N, outs[0][1])
    L2 = torch.empty_like(outs[0][0])
    N2 = torch.empty_like(outs[0][1])
    st = A.fuse_verify(x["a"].data_ptr(), x["b"].data_ptr(), x["t"].data_ptr(),
                       x["tokens"].data_ptr(), x["probs"].data_ptr(), x["unif"].data_ptr(),
                       batch.B, batch.K, batch.V, batch.dtype,
                       A.gate_params(mode=STOCH), L2.data_ptr(), N2.data_ptr(),
                       torch.cuda.current_stream().cuda_stream)
    assert st == A.OK
    torch.cuda.synchronize()
    assert torch.equal(L2, outs[0][0]) and torch.equal(N2, outs[0][1])


def test_timing_events_bracket_the_fused_row_kernel(torch):
    # the library records the caller's events around the fused row kernel only:
    # the results are unchanged and the bracketed time is positive and below the step's
    batch = small(4, 3, 40000, synth.BF16, 81)
    x = device_inputs(batch, torch)
    B, K, V = batch.B, batch.K, batch.V
    L = torch.empty(B, dtype=torch.int32, device="cuda")
    N = torch.empty_like(L)
    nbytes = A.workspace_bytes(B, K, V)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    s = torch.cuda.current_stream()
    gate = A.gate_params(mode=STOCH)
    outs = []
    for timed in (False, True):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        for e in ev:
            e.record(s)
        opts = A.LaunchOpts(0, 0, 0, 0, ev[1].cuda_event, ev[2].cuda_event) if timed else None
        assert not timed or (opts.timing_begin and opts.timing_end)
        ev[0].record(s)
        st = A.fuse_verify_ex(x["a"].data_ptr(), x["b"].data_ptr(), x["t"].data_ptr(),
                              x["tokens"].data_ptr(), x["probs"].data_ptr(), x["unif"].data_ptr(),
                              B, K, V, synth.BF16, gate, L.data_ptr(), N.data_ptr(),
                              ws.data_ptr(), nbytes, opts=opts, stream=s.cuda_stream)
        ev[3].record(s)
        assert st == A.OK
        torch.cuda.synchronize()
        outs.append((L.cpu().numpy().copy(), N.cpu().numpy().copy()))
        if timed:
            kernel_ms, step_ms = ev[1].elapsed_time(ev[2]), ev[0].elapsed_time(ev[3])
            assert 0.25 * step_ms < kernel_ms <= step_ms  # a real kernel, not two adjacent records
    assert np.array_equal(outs[0][0], outs[1][0]) and np.array_equal(outs[0][1], outs[1][1])


def test_plan_reports_cluster_occupancy(torch):
    info = A.plan(64, 7, 128256, A.BF16, opts=A.LaunchOpts(0, 0, A.KERNEL_TMA))
    assert info.kernel == A.KERNEL_TMA and info.cluster_size == 8 and info.vector_path == 1
    assert info.max_active_clusters >= 30          # 2 CTAs per SM, clusters of 8
    assert info.smem_bytes <= 113 * 1024
    info = A.plan(64, 7, 128256, A.BF16, opts=A.LaunchOpts(0, 0, A.KERNEL_GENERIC))
    assert info.kernel == A.KERNEL_GENERIC and info.max_active_clusters > 0


# ---------------------------------------------------------------- sampling law

@pytest.mark.parametrize("kernel", [GENERIC, TMA])
def test_emitted_token_law_chi_square(torch, kernel):
    from scipy.stats import chisquare
    V, K, N = 8, 1, 1_000_000
    rng = np.random.default_rng(42)
    a1 = rng.normal(0, 1, (K + 1, V)).astype(np.float32)
    b1 = (a1 + rng.normal(0, 1, (K + 1, V))).astype(np.float32)
    t1 = rng.normal(0, 1, (K + 1, V)).astype(np.float32)
    rows = [O.row_quantities(a1[k].astype(np.float64), b1[k].astype(np.float64),
                             t1[k].astype(np.float64), 0.5, 1.0, O.DIV_JSD) for k in range(K + 1)]
    p = np.exp(rows[0].la)
    d = np.minimum(np.searchsorted(np.cumsum(p), rng.uniform(0, 1, N), side="right"), V - 1)
    probs = p[d].astype(np.float32)
    unif = (rng.integers(0, 1 << 24, (N, K + 1)) / float(1 << 24)).astype(np.float32)
    batch = synth.Batch(np.broadcast_to(a1, (N, K + 1, V)), np.broadcast_to(b1, (N, K + 1, V)),
                        np.broadcast_to(t1, (N, K + 1, V)), d[:, None].astype(np.int32),
                        probs[:, None], unif, N, K, V, synth.FP32)
    g = run_gpu(batch, torch, mode=STOCH, logprobs=False, kernel=kernel, full=False)
    L, nxt = g["accept_len"], g["next_token"]
    assert np.all((L >= 0) & (L <= K)) and np.all((nxt >= 0) & (nxt < V))
    first = np.where(L >= 1, d, nxt)
    # exact law of the first emitted token (see the oracle pins)
    q = np.exp(rows[0].lq)
    A_ = np.minimum(1.0, q / (rows[0].gamma_eff * p))
    resid = np.maximum(q - p, 0.0)
    law = p * A_ + (1.0 - np.sum(p * A_)) * resid / resid.sum()
    assert chisquare(np.bincount(first, minlength=V), law * N).pvalue > 1e-3
    # and draw for draw against the oracle on the same uniforms
    oL, oN, oflag, _, _ = O.stochastic_scan(rows, d[:, None], probs[:, None].astype(np.float64),
                                            unif.astype(np.float64), K)
    ok = ~oflag
    assert ok.mean() > 0.99
    assert np.array_equal(L[ok], oL[ok]) and np.array_equal(nxt[ok], oN[ok])


@pytest.mark.parametrize("kernel", [AUTO, GENERIC])
@pytest.mark.parametrize("mode", [GREEDY, STOCH])
def test_entries_far_above_the_first_vector(torch, kernel, mode):
    # a logit 150 nats above the rest, away from every thread's first vector:
    # the fixed-reference sums overflow and the slice is redone with a
    # running maximum
    batch = small(3, 2, 40000, synth.BF16, seed=91)
    for arr in (batch.logits_full, batch.logits_comp, batch.logits_ver):
        bits = np.zeros(1, np.float32)
        bits[0] = 150.0
        spike = (bits.view(np.uint32) >> 16).astype(np.uint16)[0]
        arr[0, 1, 30001] = spike
        arr[2, 2, 12345] = spike
    for full in (False, True):
        check(batch, torch, mode, kernel, full)


# ---------------------------------------------------------------- bounded waits

@pytest.mark.parametrize("mode,full", [(GREEDY, False), (GREEDY, True), (STOCH, True)])
def test_copy_wait_timeout_marks_every_row(torch, mode, full):
    # the test hook makes every bulk-copy wait give up at once while the copies
    # still land: each CTA takes its timeout branch (marks its row, reaches every
    # cluster barrier, drains its copies before exit), and every batch element
    # comes back as a data error with ASYMSPEC_DATA_TIMEOUT; the launch returns
    # and the context stays usable (a normal call on the same inputs follows)
    batch = small(3, 2, 40000, synth.BF16, seed=17)
    x = device_inputs(batch, torch)
    fv = A.FuseVerify(batch.B, batch.K)
    res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=mode,
             row_stats=full, row_tokens=True, fused_logprobs=full, kernel=TMA,
             test_flags=A.TEST_COPY_GIVE_UP)
    torch.cuda.synchronize()
    assert list(res["accept_len"].cpu().numpy()) == [-1] * batch.B
    assert list(res["next_token"].cpu().numpy()) == [-1] * batch.B
    assert int(res["error_word"].cpu().numpy()[0]) & A.DATA_TIMEOUT
    check(batch, torch, mode, TMA, full)


def test_copy_wait_hook_ignored_by_the_production_row_kernel(torch):
    # the production row kernel waits on no copies: the hook changes nothing
    batch = small(3, 2, 40000, synth.BF16, seed=18)
    x = device_inputs(batch, torch)
    fv = A.FuseVerify(batch.B, batch.K)
    res = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=STOCH,
             kernel=TMA, test_flags=A.TEST_COPY_GIVE_UP)
    ref = fv(x["a"], x["b"], x["t"], x["tokens"], x["probs"], x["unif"], mode=STOCH, kernel=TMA)
    torch.cuda.synchronize()
    assert A.plan(3, 2, 40000, A.BF16, A.gate_params(mode=STOCH)).row_kernel == 1
    for key in ("accept_len", "next_token", "error_word"):
        assert np.array_equal(res[key].cpu().numpy(), ref[key].cpu().numpy())
    assert int(res["error_word"].cpu().numpy()[0]) == 0


# ---------------------------------------------------------------- the production row kernel

@pytest.mark.parametrize("cluster", [1, 2, 4, 5, 6, 7, 8, 10, 12, 16])
def test_row_kernel_shapes(torch, cluster):
    # the production kernel of the stochastic JSD step at every cluster size
    # the planner may take: several steps per warp, a ragged last step, bf16
    # and fp32 rows, warp blocks down to a single vector, empty warp blocks
    for B, K, V, dtype, seed in ((3, 3, 40000, synth.BF16, 61), (2, 2, 12288, synth.FP32, 62),
                                 (4, 1, 8200, synth.BF16, 63), (2, 2, 8 * cluster, synth.BF16, 64),
                                 (2, 3, 128256, synth.BF16, 65)):
        batch = small(B, K, V, dtype, seed)
        # a warp block of more than 16 steps (the decision kernel's walk loads a
        # whole block at once) is not taken by the row kernel: the staged kernel
        # takes the row if its slice fits on chip, else the planner refuses it
        vecs = -(-V // cluster) * (4 if dtype == synth.FP32 else 2) // 16
        try:
            g = run_gpu(batch, torch, mode=STOCH, full="row", cluster_size=cluster)
        except A.AsymSpecError as e:
            assert e.status == A.ERR_TOO_LARGE and vecs > 16 * 256
            continue
        info = A.plan(B, K, V, A.FP32 if dtype == synth.FP32 else A.BF16,
                      A.gate_params(mode=STOCH), A.LaunchOpts(cluster, 0, 0))
        assert info.row_kernel == (1 if vecs <= 16 * 256 else 0)
        o = run_oracle(batch, mode=STOCH, logprobs=False)
        compare(batch, g, o, mode=STOCH, logprobs=False)


def test_row_kernel_is_the_production_choice(torch):
    # clusters as small as keep the rows in flight within the L2 budget, once
    # a batch fills a wave of clusters of 8; smaller batches take 8
    for B, K, V, dtype, C in ((64, 7, 128256, A.BF16, 6), (32, 8, 151936, A.BF16, 7),
                              (8, 5, 151936, A.BF16, 8), (256, 4, 151936, A.FP32, 12),
                              (1, 4, 32000, A.FP32, 8)):
        info = A.plan(B, K, V, dtype, A.gate_params(mode=STOCH))
        assert info.kernel == A.KERNEL_TMA and info.row_kernel == 1 and info.launches == 2
        # 256-thread CTAs, four to an SM: the warps' 48 KB of load rings and the
        # cluster's pass-1 records in shared memory, no slice
        assert info.block_threads == 256 and info.cluster_size == C
        assert 4 * (info.smem_bytes + 1024) <= 228 * 1024
        assert info.max_active_clusters > 0
