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
CUDA_SRC = [os.path.join(HERE, "csrc", "asymspec.cu")]
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
    deps = list(sources) + [os.path.join(INCLUDE, "asymspec.h")]
    return any(os.path.getmtime(s) > t for s in deps)


def build_cuda(force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale(CUDA_LIB, CUDA_SRC):
        return CUDA_LIB
    tmp = CUDA_LIB + f".tmp{os.getpid()}"
    cmd = [nvcc_path(), "-gencode", GENCODE, "-O3", "-lineinfo", "-std=c++17",
           "-I" + INCLUDE, "-Xcompiler", "-fPIC", "-shared", *CUDA_SRC, "-o", tmp]
    if verbose:
        cmd.insert(1, "-Xptxas=-v")
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"nvcc failed ({' '.join(cmd)}):\n{res.stdout}\n{res.stderr}")
    if verbose:
        print(res.stderr)
    os.replace(tmp, CUDA_LIB)
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
