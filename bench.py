"""Benchmark of the fuse-and-verify step on GB300.

One step = one pass of the whole path over one batch: the C-ABI call
asymspec_fuse_verify_ex in stochastic mode (row normalisers, delta fusion,
JSD gate, acceptance tests, residual inverse-CDF draws and the per-element
accept scan): two launches, the production row kernel and the decision
kernel.  The workload is B=64, K=7, V=128256 bf16 logits with the
Zipf-profile recipe (512 verify rows, 394 MB of logits per step, larger than
the 129 MB L2; four resident input sets are rotated).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl asymspec|reference]

Under torchrun every rank runs its own replica of the workload on its own GPU
(weak scaling, no collective on the data path); rank 0 prints one JSON line.
``--impl reference`` times the float64 CPU oracle on the same workload (a
bounded sample of batch elements per step) on all the host cores.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "verify rows/s (B×(K+1) vocab rows) and achieved HBM GB/s vs GB300 peak"
WORKLOAD_CFG = 2
FALLBACK_HBM_GBS = 6800.0
CSRC = os.path.join(ROOT, "paper_2608_26004_gb300", "csrc")
KERNEL_SRCS = ("asymspec.cu", "device_common.cuh", "kernel_generic.cuh", "kernel_tma.cuh",
               "kernel_row.cuh", "kernels.h", "k_generic.cu", "k_tma_bf16.cu", "k_tma_f32.cu",
               "k_tma_bf16_prod.cu", "k_tma_f32_prod.cu", "k_tma_bf16_any_s.cu",
               "k_tma_f32_any_s.cu", "k_row_bf16.cu", "k_row_f32.cu")
N_SETS = 4          # resident input sets rotated between steps (4 x 394 MB, each > L2)
DIST_MIN_S = 1.0    # the per-step distribution loop runs at least this long
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "fuse_verify_B64_K7_V128256_bf16_traffic.txt")
REASON_BITS = {
    0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
    0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
    0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
    0x100: "display_clock_setting",
}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="asymspec", choices=["asymspec", "reference"])
    ap.add_argument("--mode", default="stochastic", choices=["stochastic", "greedy"])
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="first B batch elements only (profiling a smaller case)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_name(A, info) -> str:
    """The row kernel a call launches (the roofline's kernel)."""
    if info.kernel == A.KERNEL_TMA:
        return "fuse_verify_row" if info.row_kernel else "fuse_verify_tma"
    return "fuse_verify_generic" if info.kernel == A.KERNEL_GENERIC else str(info.kernel)


def kernel_hash() -> str:
    """sha256 (first 16 hex digits) over the kernel sources, in a fixed order."""
    h = hashlib.sha256()
    for name in KERNEL_SRCS:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def measured_traffic(mode: str):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from
    the committed ncu summary, or None once the kernel sources have changed
    since those counters were taken."""
    try:
        with open(TRAFFIC_FILE) as f:
            kv = dict(line.split(":", 1) for line in f if ":" in line and not line.startswith("#"))
    except OSError:
        return None
    kv = {k.strip(): v.strip() for k, v in kv.items()}
    if kv.get("kernel_sources_sha256_16") != kernel_hash():
        return None
    v = kv.get(f"{mode}_dram_bytes_per_launch")
    return float(v) if v else None


def algorithmic_bytes(B: int, K: int, V: int, elt: int, stochastic: bool) -> int:
    """Bytes one launch must move: every logit row it needs read once, the
    per-draft inputs, and the two int32 outputs per batch element.

    Stochastic mode needs a, b and t on all B*(K+1) rows plus the draft
    probabilities and the K+1 uniforms; greedy mode (unfused bonus) needs all
    three on the B*K draft rows but only t on the B bonus rows, and no
    probabilities or uniforms.
    """
    row = V * elt
    if stochastic:
        return 3 * row * B * (K + 1) + 4 * B * K * 2 + 4 * B * (K + 1) + 8 * B
    return 3 * row * B * K + row * B + 4 * B * K + 8 * B


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = os.path.join(tempfile.gettempdir(), f"asymspec_clocks_{os.getpid()}.csv")

    def __enter__(self):
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=index,clocks.sm,clocks.max.sm,power.draw,"
                 "clocks_event_reasons.active", "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=self.f, stderr=subprocess.DEVNULL)
            # start timing only once the sampler is producing samples
            t0 = time.time()
            while time.time() - t0 < 3.0 and os.path.getsize(self.path) == 0:
                time.sleep(0.01)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 5:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                    bits = int(parts[4], 16)
                except ValueError:
                    continue
                for b, name in REASON_BITS.items():
                    if bits & b and name != "gpu_idle":
                        reasons.add(name)
        except OSError:
            pass
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(smax)),
                "reasons": sorted(reasons), "samples": len(sm)}


def percentiles(us):
    """p10 / p50 / p90 of a list of durations (microseconds)."""
    q = np.percentile(np.asarray(us, np.float64), [10, 50, 90])
    return {"p10": float(q[0]), "p50": float(q[1]), "p90": float(q[2]), "n": len(us)}


# ---- the oracle over all host cores: one process per core (spawned), each
# generating its own copy of a bounded sample of the workload's batch elements
# at start-up, outside the timed region
_W = {}


def _oracle_init(cfg_id: int, nsample: int):
    from paper_2608_26004_gb300 import synth
    _W["batch"] = synth.make_config(cfg_id, nb=nsample)


def _oracle_element(args):
    import oracle
    b, mode_id = args
    bt = _W["batch"]
    b = b % bt.B
    sel = slice(b, b + 1)
    oracle.fuse_verify(bt.logits_full[sel], bt.logits_comp[sel], bt.logits_ver[sel],
                       bt.draft_tokens[sel], bt.draft_probs[sel], bt.uniforms[sel],
                       dtype=bt.dtype, mode=mode_id)
    return bt.K + 1


class OraclePool:
    """The float64 oracle, as it stands, run over batch elements on every host
    core (os.cpu_count() spawned processes)."""

    def __init__(self, cfg_id: int, nsample: int):
        import multiprocessing as mp
        self.cores = os.cpu_count() or 1
        self.pool = mp.get_context("spawn").Pool(self.cores, _oracle_init, (cfg_id, nsample))
        self.next = 0

    def run(self, n_elements: int, mode_id: int) -> int:
        """n_elements batch elements (cycling over the sample); returns rows done."""
        items = [(self.next + i, mode_id) for i in range(n_elements)]
        self.next += n_elements
        return sum(self.pool.map(_oracle_element, items, chunksize=1))

    def close(self):
        self.pool.close()
        self.pool.join()


def oracle_all_cores(cfg_id: int, mode_id: int, seconds: float):
    """rows/s of the oracle on all host cores for ~`seconds` (after one warm-up
    element per core)."""
    pool = OraclePool(cfg_id, nsample=16)
    try:
        pool.run(pool.cores, mode_id)
        t0 = time.perf_counter()
        rows = 0
        while time.perf_counter() - t0 < seconds:
            rows += pool.run(pool.cores, mode_id)
        el = time.perf_counter() - t0
        return rows / el, rows, el, pool.cores
    finally:
        pool.close()


def oracle_rows_per_s(batch, mode_id, seconds: float):
    """The oracle as it stands, on consecutive batch elements, for ~`seconds`."""
    import oracle
    t0 = time.perf_counter()
    rows = 0
    b = 0
    while True:
        sel = slice(b % batch.B, b % batch.B + 1)
        oracle.fuse_verify(batch.logits_full[sel], batch.logits_comp[sel], batch.logits_ver[sel],
                           batch.draft_tokens[sel], batch.draft_probs[sel], batch.uniforms[sel],
                           dtype=batch.dtype, mode=mode_id)
        rows += batch.K + 1
        b += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            return rows / el, rows, el


def draft_timing(torch, A, sets, B, K, V, mode, dev, steps):
    """Per-launch time of asymspec_draft_sample on the workload's drafter rows:
    launches of B rows (one drafted position of every batch element) and one
    launch of all B (K+1) rows, each captured K+1 (resp. 1) times per input
    set into a CUDA graph that is replayed; CUDA events around the replays."""
    rows_all = B * (K + 1)
    flat = [x["a"].view(rows_all, V) for x in sets]
    unif = [x["unif"].view(rows_all) for x in sets]
    tok = torch.empty(rows_all, dtype=torch.int32, device=dev)
    prob = torch.empty(rows_all, dtype=torch.float32, device=dev)

    def launches(rows):
        out = []
        for f, u in zip(flat, unif):
            for r0 in range(0, rows_all, rows):
                out.append((f[r0:r0 + rows], u[r0:r0 + rows]))
        return out

    def time_graph(items, rows):
        side = torch.cuda.Stream(dev)
        side.wait_stream(torch.cuda.current_stream(dev))

        def issue(stream_ptr):
            for f, u in items:
                st = A.draft_sample(f.data_ptr(), rows, V, A.BF16, mode, u.data_ptr(),
                                    tok.data_ptr(), prob.data_ptr(), 0, stream_ptr)
                if st != A.OK:
                    raise A.AsymSpecError(st, "asymspec_draft_sample")

        with torch.cuda.stream(side):
            issue(side.cuda_stream)  # warm-up, outside the graph
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            issue(side.cuda_stream)
        reps = max(3, min(200, steps))
        with torch.cuda.stream(side):
            for _ in range(3):
                g.replay()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(side)
            for _ in range(reps):
                g.replay()
            e1.record(side)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) * 1e3 / (reps * len(items))

    hbm_peak, peak_kind = peaks()
    res = {"mode": "stochastic" if mode == A.MODE_STOCHASTIC else "greedy", "kernel": "draft_kernel",
           "peak_kind": peak_kind,
           "algorithmic_bytes": "rows x V x 2 (the bf16 logits, read once) + rows x 12 "
                                "(uniform in, token and probability out)",
           "timing": "CUDA graph of the launches over both resident input sets, replayed; "
                     "CUDA events on the replay stream"}
    for key, rows in (("per_position", B), ("all_rows", rows_all)):
        us = time_graph(launches(rows), rows)
        alg = rows * V * 2 + rows * 12
        gbs = alg / (us * 1e-6) / 1e9
        res[key] = {"rows": rows, "us_per_launch": us, "hbm_gbs": gbs, "frac": gbs / hbm_peak,
                    "rows_per_s": rows / (us * 1e-6)}
    return res


def xvocab_timing(torch, A, synth, mode, dev, steps, timed, stream):
    """The cross-family step (asymspec_fuse_verify_xvocab: gather, step,
    emission) on the bench workload's batch shape over a Qwen3-sized drafter
    vocabulary, a Llama-3-sized verifier vocabulary and the paper's shared set,
    and its gather (asymspec_xvocab_gather) alone; CUDA events on the stream."""
    w = synth.CONFIGS[WORKLOAD_CFG]
    x = synth.make_xvocab(w.recipe, w.seed, w.B, w.K, synth.XVOCAB_S, synth.XVOCAB_V_D,
                          synth.XVOCAB_V_V, synth.BF16)
    B, K, S, V_d, V_v = x.B, x.K, x.S, x.V_d, x.V_v
    rows = B * (K + 1)

    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(dev)

    a, b, t = bf(x.logits_full), bf(x.logits_comp), bf(x.logits_ver)
    md = torch.from_numpy(x.map_d).to(dev)
    mv = torch.from_numpy(x.map_v).to(dev)
    d = torch.from_numpy(x.draft_tokens).to(dev)
    pr = torch.from_numpy(x.draft_probs).to(dev)
    u = torch.from_numpy(x.uniforms).to(dev)
    nbytes = A.xvocab_workspace_bytes(B, K, S, V_d, V_v, A.BF16)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    L = torch.empty(B, dtype=torch.int32, device=dev)
    N = torch.empty(B, dtype=torch.int32, device=dev)
    gate = A.gate_params(mode=mode)
    sptr = stream.cuda_stream

    def step(i):
        st = A.fuse_verify_xvocab(a.data_ptr(), b.data_ptr(), V_d, t.data_ptr(), V_v,
                                  md.data_ptr(), mv.data_ptr(), S, d.data_ptr(), pr.data_ptr(),
                                  u.data_ptr(), B, K, A.BF16, gate, L.data_ptr(), N.data_ptr(),
                                  0, ws.data_ptr(), nbytes, None, sptr)
        if st != A.OK:
            raise A.AsymSpecError(st, "asymspec_fuse_verify_xvocab")

    g_out = torch.empty(3, rows, S, dtype=torch.bfloat16, device=dev)
    sc_n = A.xvocab_gather_scratch_bytes(V_d, V_v)
    sc = torch.empty(sc_n, dtype=torch.uint8, device=dev)

    def gather(i):
        st = A.xvocab_gather(a.data_ptr(), b.data_ptr(), V_d, t.data_ptr(), V_v, md.data_ptr(),
                             mv.data_ptr(), S, rows, A.BF16, g_out[0].data_ptr(),
                             g_out[1].data_ptr(), g_out[2].data_ptr(), None, sc.data_ptr(), sc_n,
                             sptr)
        if st != A.OK:
            raise A.AsymSpecError(st, "asymspec_xvocab_gather")

    n = max(3, min(steps, 50))
    ms_step = timed(step, n, 3) / n
    ms_gather = timed(gather, n, 3) / n
    del g_out, ws

    # the gather must bring in every 32-byte DRAM sector holding a paired entry
    # and write the restricted rows densely
    def sectors(m):
        return int(np.unique(m.astype(np.int64) * 2 // 32).size)

    touched = rows * 32 * (2 * sectors(x.map_d) + sectors(x.map_v))
    written = rows * 3 * S * 2
    hbm_peak, peak_kind = peaks()
    g_gbs = (touched + written) / (ms_gather * 1e-3) / 1e9
    return {"mode": "stochastic" if mode == A.MODE_STOCHASTIC else "greedy",
            "B": B, "K": K, "S": S, "V_d": V_d, "V_v": V_v, "rows": rows,
            "ms_per_step": ms_step, "rows_per_s": rows / (ms_step * 1e-3),
            "launches_per_step": 6,
            "gather": {"kernel": "xvocab_gather", "us_per_launch": ms_gather * 1e3,
                       "algorithmic_bytes_per_launch": touched + written,
                       "algorithmic_bytes": "the 32-byte sectors of a, b and t holding paired "
                                            "entries, read once, plus the restricted rows "
                                            "written once (the inverse maps the launch builds "
                                            "and reads are not counted)",
                       "launches": "the map check (inverse-map fill and build), then the gather",
                       "hbm_gbs": g_gbs, "frac": g_gbs / hbm_peak, "peak_kind": peak_kind},
            "timing": "CUDA events around the timed calls on the launching stream"}


def max_over_ranks(ms: float, dist=None, device="cpu") -> float:
    """The slowest rank's time: an all-reduce MAX over the process group (the
    value itself with a single process)."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_rows_per_s(world: int, rows_per_rank: int, ms_per_step: float) -> float:
    """Whole-job throughput: every rank verifies its own rows_per_rank rows per
    step (replicas, weak scaling), in the slowest rank's step time."""
    return world * rows_per_rank / (ms_per_step * 1e-3)


def run_reference(args, workload, rank, world):
    """--impl reference: the float64 CPU oracle, timed on all the host cores
    (one batch element per core per step)."""
    if rank != 0:
        return
    mode_id = 1 if args.mode == "stochastic" else 0
    pool = OraclePool(WORKLOAD_CFG, nsample=16)
    try:
        for _ in range(max(args.warmup, 1)):
            pool.run(pool.cores, mode_id)
        t0 = time.perf_counter()
        rows = 0
        for _ in range(args.steps):
            rows += pool.run(pool.cores, mode_id)
        el = time.perf_counter() - t0
    finally:
        pool.close()
    value = rows / el
    sample = (f"each step: {pool.cores} batch elements (one per host core; K+1={workload.K + 1} "
              f"rows of V={workload.V} each) cycling over the first 16 elements of "
              f"{workload.name}, float64 numpy oracle, {pool.cores} processes")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "rows/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * el / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload.name, "B": workload.B, "K": workload.K,
                   "V": workload.V, "logits": "bf16", "mode": args.mode},
        "cpu_baseline": {"value": value, "unit": "rows/s", "cores": pool.cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    rank, world, local = dist_env()
    from paper_2608_26004_gb300 import synth
    workload = synth.CONFIGS[WORKLOAD_CFG]
    if args.impl == "reference":
        run_reference(args, workload, rank, world)
        return

    import torch
    from paper_2608_26004_gb300 import asymspec as A

    assert torch.cuda.is_available(), "bench.py needs a CUDA device"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist

    mode = A.MODE_STOCHASTIC if args.mode == "stochastic" else A.MODE_GREEDY
    batch = synth.make_config(WORKLOAD_CFG, nb=args.batch or None)
    B, K, V = batch.B, batch.K, batch.V
    rows = B * (K + 1)
    alg_bytes = algorithmic_bytes(B, K, V, 2, mode == A.MODE_STOCHASTIC)

    def to_dev_logits(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).to(dev)

    sets = []
    for rep in range(N_SETS):  # resident input sets, rotated (each larger than L2)
        sets.append(dict(
            a=to_dev_logits(batch.logits_full), b=to_dev_logits(batch.logits_comp),
            t=to_dev_logits(batch.logits_ver),
            tok=torch.from_numpy(batch.draft_tokens).to(dev),
            prob=torch.from_numpy(batch.draft_probs).to(dev),
            unif=torch.from_numpy(batch.uniforms).to(dev)))
    L = torch.empty(B, dtype=torch.int32, device=dev)
    N = torch.empty(B, dtype=torch.int32, device=dev)
    nbytes = A.workspace_bytes(B, K, V)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    gate = A.gate_params(mode=mode)
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream
    info = A.plan(B, K, V, A.BF16, gate)

    def step(x, opts=None):
        st = A.fuse_verify_ex(x["a"].data_ptr(), x["b"].data_ptr(), x["t"].data_ptr(),
                              x["tok"].data_ptr(), x["prob"].data_ptr(), x["unif"].data_ptr(),
                              B, K, V, A.BF16, gate, L.data_ptr(), N.data_ptr(), ws.data_ptr(),
                              nbytes, opts=opts, stream=sptr)
        if st != A.OK:
            raise A.AsymSpecError(st, "asymspec_fuse_verify_ex")

    # the per-step distribution loop: events around every step, and the events
    # the library records around the fused row kernel of every step
    # (asymspec_launch_opts.timing_begin / timing_end), all on the one stream.
    # It runs at least DIST_MIN_S seconds (so that the clock sampler sees it).
    n_dist = max(args.steps, 64)
    sev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(n_dist)]
    kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(n_dist)]
    for b, e in kev + sev:  # torch creates an event at its first record: before taking handles
        b.record(stream)
        e.record(stream)
    kopts = [A.LaunchOpts(0, 0, 0, 0, b.cuda_event, e.cuda_event) for b, e in kev]
    assert all(o.timing_begin and o.timing_end for o in kopts)

    def timed(fn, steps, warmup):
        for i in range(warmup):
            fn(i)
        torch.cuda.synchronize(dev)
        if pg:
            pg.barrier()
        torch.cuda.synchronize(dev)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(steps):
            fn(i)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        if pg:
            pg.barrier()
        torch.cuda.synchronize(dev)
        return max_over_ranks(e0.elapsed_time(e1), pg, dev)

    def dist_step(i):
        j = i % n_dist
        sev[j][0].record(stream)
        step(sets[i % N_SETS], kopts[j])
        sev[j][1].record(stream)

    # ---- device-resident throughput (the headline value)
    with ClockSampler(local) as clk:
        ms = timed(lambda i: step(sets[i % N_SETS]), args.steps, max(args.warmup, 3))
        # the distribution loop (kept out of the headline loop: the records add
        # a few us a step): per-step and per-kernel events, repeated until it
        # has run DIST_MIN_S seconds; the last pass's events are kept
        step_us, kern_us, t0 = [], [], time.time()
        while True:
            timed(dist_step, n_dist, max(args.warmup, 3))
            step_us = [1e3 * b.elapsed_time(e) for b, e in sev]
            kern_us = [1e3 * b.elapsed_time(e) for b, e in kev]
            if time.time() - t0 >= DIST_MIN_S:
                break
    clocks = clk.summary()
    ms_step = ms / args.steps
    value = aggregate_rows_per_s(world, rows, ms_step)
    # the roofline is the fused row kernel's own: its mean duration between
    # the events the library recorded around it in every step of the
    # distribution loop (the decision kernel that follows it is not included)
    launches_per_step = info.launches
    kernel_ms = float(np.mean(kern_us)) * 1e-3
    launch_s = kernel_ms * 1e-3
    hbm_peak, peak_kind = peaks()
    achieved = alg_bytes / launch_s / 1e9

    # ---- the other mode, same workload (reported alongside)
    other_mode = A.MODE_GREEDY if mode == A.MODE_STOCHASTIC else A.MODE_STOCHASTIC
    gate_o = A.gate_params(mode=other_mode)

    def step_o(x):
        st = A.fuse_verify_ex(x["a"].data_ptr(), x["b"].data_ptr(), x["t"].data_ptr(),
                              x["tok"].data_ptr(), x["prob"].data_ptr(), x["unif"].data_ptr(),
                              B, K, V, A.BF16, gate_o, L.data_ptr(), N.data_ptr(), ws.data_ptr(),
                              nbytes, stream=sptr)
        if st != A.OK:
            raise A.AsymSpecError(st, "asymspec_fuse_verify_ex")

    ms_o = timed(lambda i: step_o(sets[i % N_SETS]), args.steps, max(args.warmup, 3)) / args.steps

    alg_bytes_o = algorithmic_bytes(B, K, V, 2, other_mode == A.MODE_STOCHASTIC)

    # ---- end to end through the C ABI with host buffers
    pin = dict(
        a=torch.from_numpy(np.ascontiguousarray(batch.logits_full).view(np.int16)).view(
            torch.bfloat16).pin_memory(),
        b=torch.from_numpy(np.ascontiguousarray(batch.logits_comp).view(np.int16)).view(
            torch.bfloat16).pin_memory(),
        t=torch.from_numpy(np.ascontiguousarray(batch.logits_ver).view(np.int16)).view(
            torch.bfloat16).pin_memory(),
        tok=torch.from_numpy(batch.draft_tokens).pin_memory(),
        prob=torch.from_numpy(batch.draft_probs).pin_memory(),
        unif=torch.from_numpy(batch.uniforms).pin_memory())
    hL = torch.empty(B, dtype=torch.int32).pin_memory()
    hN = torch.empty(B, dtype=torch.int32).pin_memory()
    h2d = sum(v.numel() * v.element_size() for v in pin.values())
    d2h = 2 * B * 4
    # asymspec_fuse_verify_host: the public call with host buffers, its copies
    # pipelined with the kernels in chunks of batch elements
    sbytes = A.host_scratch_bytes(B, K, V, A.BF16)
    scratch = torch.empty(sbytes, dtype=torch.uint8, device=dev)

    def e2e_step(i):
        st = A.fuse_verify_host(pin["a"].data_ptr(), pin["b"].data_ptr(), pin["t"].data_ptr(),
                                pin["tok"].data_ptr(), pin["prob"].data_ptr(),
                                pin["unif"].data_ptr(), B, K, V, A.BF16, gate, hL.data_ptr(),
                                hN.data_ptr(), scratch.data_ptr(), sbytes, sptr)
        if st != A.OK:
            raise A.AsymSpecError(st, "asymspec_fuse_verify_host")

    e2e_steps = max(3, min(args.steps, 30))
    ms_e2e = timed(e2e_step, e2e_steps, 3) / e2e_steps
    e2e_value = aggregate_rows_per_s(world, rows, ms_e2e)

    # ---- the drafter's draw (asymspec_draft_sample), the step upstream of
    # fuse-and-verify: per drafted position one launch over the B rows of the
    # drafter's full-context logits, and once over all B (K+1) rows.  Timed as
    # CUDA graph replays (host launch overhead would exceed a 64-row launch);
    # the launches read the rows of both resident sets in turn (262 MB > L2).
    draft = draft_timing(torch, A, sets, B, K, V, mode, dev, args.steps)

    # ---- the cross-family step (drafter and verifier vocabularies that
    # differ, restricted to their shared tokens): reported alongside
    xvocab = xvocab_timing(torch, A, synth, mode, dev, args.steps, timed, stream)


    line = {
        "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": workload.name if B == workload.B else f"{workload.name}_first{B}",
                   "B": B, "K": K, "V": V, "logits": "bf16",
                   "mode": args.mode, "rows_per_gpu": rows, "gamma": 0.5, "beta": 1.0,
                   "divergence": "jsd",
                   "l2": f"inputs larger than L2: {N_SETS} resident sets of "
                         f"{3 * rows * V * 2 / 1e6:.0f} MB rotated",
                   "cluster_size": info.cluster_size, "ctas": info.ctas,
                   "parallelism": f"replicas x{world}"},
        "hbm_gbs": achieved,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "peak_kind": peak_kind,
                     "traffic": measured_traffic(args.mode),
                     "algorithmic_bytes_per_launch": alg_bytes,
                     "kernel": kernel_name(A, info),
                     "launch_us": kernel_ms * 1e3,
                     "launch_us_pct": percentiles(kern_us),
                     "timing": "CUDA events the library records around the fused row kernel "
                               f"on its stream, in every step of a loop of {n_dist} steps "
                               "(repeated until it has run 1 s; the last pass is kept), "
                               "separate from the headline loop"},
        "step_us_pct": percentiles(step_us),
        "e2e": {"value": e2e_value, "unit": "rows/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
        "draft": draft,
        "xvocab": xvocab,
        "other_mode": {"mode": "greedy" if other_mode == A.MODE_GREEDY else "stochastic",
                       "ms_per_step": ms_o, "rows_per_s": world * rows / (ms_o * 1e-3),
                       "hbm_gbs": alg_bytes_o / (ms_o * 1e-3) / 1e9,
                       "algorithmic_bytes_per_launch": alg_bytes_o,
                       "traffic": measured_traffic(
                           "greedy" if other_mode == A.MODE_GREEDY else "stochastic")},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        mode_id = 1 if mode == A.MODE_STOCHASTIC else 0
        rps, nrows, el, cores = oracle_all_cores(WORKLOAD_CFG, mode_id, args.cpu_seconds)
        rps1, nrows1, el1 = oracle_rows_per_s(batch, mode_id, args.cpu_seconds)
        line["cpu_baseline"] = {
            "value": rps, "unit": "rows/s", "cores": cores, "kind": "oracle",
            "sample": f"{nrows} rows ({nrows // (K + 1)} batch elements, cycling over the first "
                      f"16) of {workload.name} in {el:.1f} s, float64 numpy oracle, one "
                      f"process per host core ({cores})",
            "single_thread": {
                "value": rps1, "unit": "rows/s", "cores": 1,
                "sample": f"{nrows1} rows ({nrows1 // (K + 1)} batch elements) of "
                          f"{workload.name} in {el1:.1f} s, float64 numpy oracle, one thread"}}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
