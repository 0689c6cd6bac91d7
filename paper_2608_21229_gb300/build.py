"""Build the CUDA library (librefcache.so) for sm_103a with nvcc, in-tree.

The library is one translation unit (csrc/refcache.cu, which includes the
kernels) compiled with ``-gencode arch=compute_103a,code=sm_103a`` and linked
against the shared CUDA runtime, so that it shares the runtime (and the
streams) of the host process.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "librefcache.so")
ARCH_FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a"]


def cuda_home() -> str:
    for c in (os.environ.get("CUDA_HOME"), os.environ.get("CUDA_PATH"), "/usr/local/cuda"):
        if c and os.path.exists(os.path.join(c, "bin", "nvcc")):
            return c
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    raise RuntimeError("nvcc not found: set CUDA_HOME")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cu", ".cuh", ".h"))) + [
        os.path.join(INCLUDE, "refcache.h")]


def up_to_date() -> bool:
    if not os.path.exists(LIB_PATH):
        return False
    t = os.path.getmtime(LIB_PATH)
    return all(os.path.getmtime(s) <= t for s in sources())


def nvcc_cmd(out: str, extra=()) -> list:
    home = cuda_home()
    return [
        os.path.join(home, "bin", "nvcc"), *ARCH_FLAGS, "-O3", "-lineinfo", "-std=c++17", "-shared",
        "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden", "--expt-relaxed-constexpr",
        "-cudart", "shared", f"-I{INCLUDE}", f"-I{CSRC}", os.path.join(CSRC, "refcache.cu"),
        "-o", out, f"-L{os.path.join(home, 'lib64')}", f"-Xlinker", f"-rpath={os.path.join(home, 'lib64')}",
        *extra,
    ]


def build(force: bool = False, verbose: bool = False, extra=()) -> str:
    if not force and not extra and up_to_date():
        return LIB_PATH
    os.makedirs(BUILD_DIR, exist_ok=True)
    tmp = LIB_PATH + f".tmp{os.getpid()}"
    cmd = nvcc_cmd(tmp, extra)
    if verbose:
        print(" ".join(cmd), file=sys.stderr)
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True,
          extra=["-Xptxas", "-v"] if "--ptxas-v" in sys.argv else ())
