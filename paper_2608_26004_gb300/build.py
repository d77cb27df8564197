"""Builds the native libraries in place (no cmake, no setuptools).

* ``libasymspec.so``: the sm_103a kernels and the C ABI of include/asymspec.h,
  compiled with nvcc for ``-gencode arch=compute_103a,code=sm_103a`` only.
* ``libasymspec_synth.so``: the host input generator (plain C, gcc).
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
INCLUDE = os.path.join(ROOT, "include")
CSRC = os.path.join(HERE, "csrc")
# one translation unit per kernel family and dtype, compiled in parallel
CUDA_SRC = [os.path.join(CSRC, f) for f in (
    "asymspec.cu", "k_generic.cu", "k_tma_bf16.cu", "k_tma_f32.cu", "k_tma_bf16_prod.cu",
    "k_tma_f32_prod.cu", "k_tma_bf16_any_s.cu", "k_tma_f32_any_s.cu", "k_row_bf16.cu",
    "k_row_f32.cu", "k_draft.cu", "k_xvocab.cu")]
CUDA_HEADERS = [os.path.join(CSRC, f) for f in (
    "device_common.cuh", "kernel_generic.cuh", "kernel_tma.cuh", "kernel_row.cuh",
    "kernel_draft.cuh", "kernel_xvocab.cuh", "kernels.h")]
CUDA_LIB = os.path.join(HERE, "libasymspec.so")
GENCODE = "arch=compute_103a,code=sm_103a"


def nvcc_path() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libasymspec.so")


def _stale(target: str, sources) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    deps = list(sources) + CUDA_HEADERS + [os.path.join(INCLUDE, "asymspec.h")]
    return any(os.path.getmtime(s) > t for s in deps)


def _run(cmd):
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"nvcc failed ({' '.join(cmd)}):\n{res.stdout}\n{res.stderr}")
    return res.stderr


def build_cuda(force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale(CUDA_LIB, CUDA_SRC):
        return CUDA_LIB
    nvcc = nvcc_path()
    tag = f".tmp{os.getpid()}"
    objs = [os.path.join(CSRC, os.path.basename(src)[:-3] + tag + ".o") for src in CUDA_SRC]
    base = [nvcc, "-gencode", GENCODE, "-O3", "-lineinfo", "-std=c++17", "-I" + INCLUDE,
            "-Xcompiler", "-fPIC"]
    if verbose:
        base.append("-Xptxas=-v")
    try:
        with ThreadPoolExecutor(len(CUDA_SRC)) as ex:
            logs = list(ex.map(_run, [base + ["-c", src, "-o", obj]
                                      for src, obj in zip(CUDA_SRC, objs)]))
        tmp = CUDA_LIB + tag
        _run([nvcc, "-shared", "-gencode", GENCODE, *objs, "-o", tmp])
        os.replace(tmp, CUDA_LIB)
    finally:
        for obj in objs:
            if os.path.exists(obj):
                os.remove(obj)
    if verbose:
        print("".join(logs))
    return CUDA_LIB


def build_all(force: bool = False, verbose: bool = False) -> None:
    from . import synth
    with ThreadPoolExecutor(2) as ex:
        f1 = ex.submit(build_cuda, force, verbose)
        f2 = ex.submit(synth.build, force)
        f1.result()
        f2.result()


if __name__ == "__main__":
    build_all(force=True, verbose=True)
