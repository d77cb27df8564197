"""Seeded synthetic inputs shaped like the paper's verifier and drafter vocabularies.

The five workloads below stand in for the logits of the paper's models
(Qwen3 vocabularies of 151,936 tokens and Llama-3 vocabularies of 128,256
tokens, Section 4.2 and Appendix C) and its datasets, none of which are used.
Each row triple is (drafter on the full context ``a``, drafter on the
compressed context ``b``, verifier on the compressed context ``t``), the three
forward passes of Section 3.2.

The arithmetic lives in ``csrc/synth.c`` (Philox4x32-10 counters, Box-Muller
normals); this module only describes the recipes and marshals buffers.  It
holds none of the fuse-and-verify arithmetic and is shared by the oracle tests,
the GPU tests and the benchmark.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "csrc", "synth.c")
_LIB = os.path.join(_HERE, "libasymspec_synth.so")

FP32 = 0
BF16 = 1


class _Recipe(ctypes.Structure):
    _fields_ = [
        ("profile", ctypes.c_int),
        ("sigma_v", ctypes.c_double),
        ("spike", ctypes.c_double),
        ("zipf_s", ctypes.c_double),
        ("zipf_noise", ctypes.c_double),
        ("sigma_f", ctypes.c_double),
        ("frac_lo", ctypes.c_double),
        ("frac_hi", ctypes.c_double),
        ("sigma_c", ctypes.c_double),
        ("identical_lower_half", ctypes.c_int),
    ]


@dataclass(frozen=True)
class Recipe:
    """Generative recipe of one workload (all scales are standard deviations)."""

    profile: int = 0  # 0: N(0, sigma_v^2) plus a spike on one token; 1: Zipf profile
    sigma_v: float = 2.0
    spike: float = 8.0
    zipf_s: float = 1.1
    zipf_noise: float = 0.3
    sigma_f: float = 0.5
    frac_lo: float = 0.05
    frac_hi: float = 0.05
    sigma_c: float = 3.0
    identical_lower_half: bool = False

    def _c(self) -> _Recipe:
        return _Recipe(self.profile, self.sigma_v, self.spike, self.zipf_s,
                       self.zipf_noise, self.sigma_f, self.frac_lo, self.frac_hi,
                       self.sigma_c, int(self.identical_lower_half))


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    K: int
    V: int
    dtype: int
    recipe: Recipe
    seed: int
    sweep: tuple = field(default=())  # perturbation scales for the divergence sweep


def _seed(cfg_id: int) -> int:
    return 0xA5A50000 + cfg_id


# The five workloads.  Scales not stated in the workload descriptions are
# chosen as follows: config 2 perturbs by N(0, 3^2) like config 0; config 4
# perturbs 5% of tokens at each sweep scale.
CONFIGS = {
    0: Workload("B1_K4_V32000_fp32", 1, 4, 32000, FP32,
                Recipe(frac_lo=0.05, frac_hi=0.05, sigma_c=3.0), _seed(0)),
    1: Workload("B8_K5_V151936_bf16", 8, 5, 151936, BF16,
                Recipe(frac_lo=0.02, frac_hi=0.02, sigma_c=2.0), _seed(1)),
    2: Workload("B64_K7_V128256_bf16_zipf", 64, 7, 128256, BF16,
                Recipe(profile=1, frac_lo=0.0, frac_hi=0.10, sigma_c=3.0), _seed(2)),
    3: Workload("B256_K4_V151936_fp32", 256, 4, 151936, FP32,
                Recipe(frac_lo=0.20, frac_hi=0.20, sigma_c=4.0,
                       identical_lower_half=True), _seed(3)),
    4: Workload("B32_K8_V151936_bf16_sweep", 32, 8, 151936, BF16,
                Recipe(frac_lo=0.05, frac_hi=0.05, sigma_c=0.0), _seed(4),
                sweep=(0.0, 0.5, 1.0, 2.0, 4.0, 8.0)),
}


def build(force: bool = False) -> str:
    """Compiles the host generator into a shared library next to this file."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
               "-fPIC", "-shared", "-pthread", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.asymspec_synth_generate.restype = ctypes.c_int
        lib.asymspec_synth_generate.argtypes = [
            ctypes.POINTER(_Recipe), ctypes.c_uint64, ctypes.c_int, ctypes.c_int,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int]
        lib.asymspec_philox4x32_10.restype = None
        lib.asymspec_philox4x32_10.argtypes = [
            ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_uint32),
            ctypes.POINTER(ctypes.c_uint32)]
        _lib = lib
    return _lib


def philox4x32_10(ctr, key):
    """One Philox4x32-10 block (exposed so tests can pin the generator)."""
    lib = _load()
    c = (ctypes.c_uint32 * 4)(*ctr)
    k = (ctypes.c_uint32 * 2)(*key)
    o = (ctypes.c_uint32 * 4)()
    lib.asymspec_philox4x32_10(c, k, o)
    return tuple(int(x) for x in o)


@dataclass
class Batch:
    """Host arrays of one workload (bf16 logits are uint16 bit patterns)."""

    logits_full: np.ndarray
    logits_comp: np.ndarray
    logits_ver: np.ndarray
    draft_tokens: np.ndarray
    draft_probs: np.ndarray
    uniforms: np.ndarray
    B: int
    K: int
    V: int
    dtype: int
    b0: int = 0

    @property
    def rows(self) -> int:
        return self.B * (self.K + 1)

    @property
    def logit_bytes(self) -> int:
        return 3 * self.rows * self.V * (2 if self.dtype == BF16 else 4)


def bf16_bits_to_f32(u16: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (u16.astype(np.uint32) << 16).view(np.float32)


def generate(recipe: Recipe, seed: int, B: int, K: int, V: int, dtype: int,
             b0: int = 0, nb: int | None = None, B_total: int | None = None,
             nthreads: int = 0) -> Batch:
    """Generates batch elements [b0, b0+nb) of a workload with B_total elements."""
    if nb is None:
        nb = B - b0
    if B_total is None:
        B_total = B
    if nthreads <= 0:
        nthreads = min(os.cpu_count() or 1, 32)
    lib = _load()
    ldt = np.float32 if dtype == FP32 else np.uint16
    shape = (nb, K + 1, V)
    full = np.empty(shape, ldt)
    comp = np.empty(shape, ldt)
    ver = np.empty(shape, ldt)
    tokens = np.empty((nb, K), np.int32)
    probs = np.empty((nb, K), np.float32)
    unif = np.empty((nb, K + 1), np.float32)
    rc = recipe._c()
    ret = lib.asymspec_synth_generate(
        ctypes.byref(rc), seed, b0, nb, B_total, K, V, dtype,
        full.ctypes.data, comp.ctypes.data, ver.ctypes.data, tokens.ctypes.data,
        probs.ctypes.data, unif.ctypes.data, nthreads)
    if ret != 0:
        raise RuntimeError(f"asymspec_synth_generate failed with {ret}")
    return Batch(full, comp, ver, tokens, probs, unif, nb, K, V, dtype, b0)


def make_config(cfg_id: int, sweep_index: int = 0, b0: int = 0, nb: int | None = None,
                nthreads: int = 0) -> Batch:
    """Batch elements [b0, b0+nb) of one of the five workloads."""
    w = CONFIGS[cfg_id]
    rc = w.recipe
    if w.sweep:
        rc = Recipe(**{**rc.__dict__, "sigma_c": w.sweep[sweep_index]})
    if nb is None:
        nb = w.B - b0
    return generate(rc, w.seed, w.B, w.K, w.V, w.dtype, b0=b0, nb=nb, B_total=w.B,
                    nthreads=nthreads)


# ------------------------------------------------- cross-family vocabularies

# The paper's heterogeneous pairings (Section 4, "Cross-family portability")
# share 109,566 string-identical tokens plus paired special tokens between a
# Qwen3 (151,936) and a Llama-3 (128,256) vocabulary; two special pairs are
# taken here, which makes S = 109,568.
XVOCAB_S = 109_568
XVOCAB_V_D = 151_936
XVOCAB_V_V = 128_256


@dataclass
class XBatch:
    """A step whose drafter (vocabulary V_d) and verifier (vocabulary V_v)
    share S tokens, the pairs (map_d[j], map_v[j]).  logits_full and
    logits_comp are [B, K+1, V_d], logits_ver [B, K+1, V_v]; draft_tokens are
    pair indices in [0, S) and draft_probs their probabilities under the
    drafter's softmax over the pairs."""

    logits_full: np.ndarray
    logits_comp: np.ndarray
    logits_ver: np.ndarray
    map_d: np.ndarray
    map_v: np.ndarray
    draft_tokens: np.ndarray
    draft_probs: np.ndarray
    uniforms: np.ndarray
    B: int
    K: int
    S: int
    V_d: int
    V_v: int
    dtype: int


def _f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even bf16 bit patterns of finite float32 values."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32)
    return ((u + (((u >> 16) & 1) + 0x7FFF)) >> 16).astype(np.uint16)


def make_xvocab(recipe: Recipe, seed: int, B: int, K: int, S: int, V_d: int, V_v: int,
                dtype: int, unpaired_mean: float = 3.0, nthreads: int = 0) -> XBatch:
    """Cross-family inputs: the workload recipe generated over the S shared
    tokens (so the drafts and their probabilities are those of the shared
    set), scattered into the two vocabularies through a seeded map.  map_d
    is an increasing subset of the drafter's tokens, map_v a random
    injection into the verifier's; the unpaired logits are N(unpaired_mean,
    2^2), above the paired ones on average, so that a path that read them
    would visibly change every normaliser."""
    if not (2 <= S <= min(V_d, V_v)):
        raise ValueError("need 2 <= S <= min(V_d, V_v)")
    inner = generate(recipe, seed, B, K, S, dtype, nthreads=nthreads)
    rng = np.random.default_rng(seed)
    map_d = np.sort(rng.choice(V_d, S, replace=False)).astype(np.int32)
    map_v = rng.choice(V_v, S, replace=False).astype(np.int32)

    def scatter(rows, V, idx):
        fill = rng.normal(unpaired_mean, 2.0, (B, K + 1, V)).astype(np.float32)
        out = fill if dtype == FP32 else _f32_to_bf16_bits(fill)
        out[..., idx] = rows
        return out

    return XBatch(scatter(inner.logits_full, V_d, map_d), scatter(inner.logits_comp, V_d, map_d),
                  scatter(inner.logits_ver, V_v, map_v), map_d, map_v, inner.draft_tokens,
                  inner.draft_probs, inner.uniforms, B, K, S, V_d, V_v, dtype)
