"""Builds the CUDA library in-tree: libgnn_gb300.so next to this file.

nvcc, sm_103a only; the C++ runtime is linked statically into the library so
the shared object has no dependency beyond the CUDA driver."""
from __future__ import annotations

import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
LIB = os.path.join(HERE, "libgnn_gb300.so")
SOURCES = [os.path.join(HERE, "csrc", "gnn_api.cu")]
DEPS = SOURCES + [os.path.join(HERE, "csrc", f) for f in ("ptx.cuh", "csr.cuh", "mlp_tiles.cuh", "components.cuh", "compact.cuh", "frnn.cuh")] + \
    [os.path.join(ROOT, "include", "gnn.h")]
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")
FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo", "-std=c++17",
         "-Xcompiler", "-fPIC", "-shared", "--expt-relaxed-constexpr", "-cudart", "static"]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(d) <= t for d in DEPS)


def build(force: bool = False, verbose: bool = False, extra=()) -> str:
    if force or not up_to_date():
        cmd = [NVCC, *FLAGS, *extra, "-o", LIB + ".tmp", *SOURCES]
        if verbose:
            print(" ".join(cmd), file=sys.stderr)
        subprocess.run(cmd, check=True)
        os.replace(LIB + ".tmp", LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True,
          extra=["-Xptxas", "-v"] if "--ptxas" in sys.argv else [])
