"""Compile libautoverse.so in-tree for sm_103a (nvcc, no cmake)."""
from __future__ import annotations

import os
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
LIB = os.path.join(PKG, "libautoverse.so")
SOURCES = [os.path.join(CSRC, f) for f in ("autoverse.cu", "k_fast_u8.cu", "k_fast_u16.cu", "k_warp_u8.cu",
                                            "k_warp_u16.cu", "k_block.cu", "k_expand.cu", "k_search.cu",
                                            "k_observe.cu", "k_mutate.cu", "k_memo_u8.cu", "k_memo_u16.cu",
                                            "k_variant.cu", "k_band.cu", "k_step.cu")]
DEPS = SOURCES + [os.path.join(CSRC, f) for f in ("kernels.cuh", "launch.h", "k_fast_impl.cuh", "k_warp_impl.cuh",
                                                     "k_memo_impl.cuh")] + [
    os.path.join(ROOT, "include", "autoverse.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def build(force: bool = False, verbose: bool = False, extra: list | None = None) -> str:
    """Build the shared library next to this file: every translation unit is
    compiled in parallel, then linked.  Returns the library's path."""
    stale = not os.path.exists(LIB) or any(os.path.getmtime(d) > os.path.getmtime(LIB) for d in DEPS)
    if not (force or stale or extra):
        return LIB
    import tempfile
    from concurrent.futures import ThreadPoolExecutor
    cuda_lib = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "lib64")
    common = [nvcc(), "-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-lineinfo", *ARCH,
              "-I", os.path.join(ROOT, "include"), *(extra or [])]
    with tempfile.TemporaryDirectory() as tmpdir:
        objs = [os.path.join(tmpdir, os.path.basename(src) + ".o") for src in SOURCES]
        cmds = [common + ["-c", src, "-o", obj] for src, obj in zip(SOURCES, objs)]
        if verbose:
            for cmd in cmds:
                print(" ".join(cmd))
        with ThreadPoolExecutor(max_workers=len(cmds)) as pool:
            list(pool.map(subprocess.check_call, cmds))
        tmp = LIB + f".tmp{os.getpid()}"
        link = [nvcc(), "-shared", *ARCH, "-cudart", "shared", "-Xlinker", "-rpath", "-Xlinker", cuda_lib,
                *objs, "-o", tmp]
        if verbose:
            print(" ".join(link))
        subprocess.check_call(link)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(force=True, verbose=True)
