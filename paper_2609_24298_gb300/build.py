"""Build libcobra.so in-tree for sm_103a (nvcc; host code through nvcc's host compiler).

The host allocator is compiled without floating-point contraction so its results are
reproducible bit for bit (see csrc/host.cpp)."""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libcobra.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")


def _run(cmd):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        sys.stderr.write(r.stdout + r.stderr)
        raise RuntimeError("command failed: " + " ".join(cmd))
    return r.stdout + r.stderr


def build(verbose: bool = False) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    common = ["-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-ffp-contract=off", "-I", CSRC]
    jobs = [
        [NVCC, *ARCH, *common, "-x", "cu", "-c", os.path.join(CSRC, "host.cpp"), "-o", os.path.join(OUT_DIR, "host.o")],
        [NVCC, *ARCH, *common, "-lineinfo", "-Xptxas", "-v", "-c", os.path.join(CSRC, "kernels.cu"), "-o",
         os.path.join(OUT_DIR, "kernels.o")],
    ]
    with ThreadPoolExecutor(len(jobs)) as ex:
        logs = list(ex.map(_run, jobs))
    if verbose:
        for l in logs:
            sys.stderr.write(l)
    _run([NVCC, *ARCH, "-shared", "-o", LIB, os.path.join(OUT_DIR, "host.o"), os.path.join(OUT_DIR, "kernels.o"),
          "-lcudart"])
    with open(os.path.join(OUT_DIR, "ptxas.log"), "w") as f:
        f.write("\n".join(logs))
    return LIB


if __name__ == "__main__":
    build(verbose="-v" in sys.argv)
    print(LIB)
