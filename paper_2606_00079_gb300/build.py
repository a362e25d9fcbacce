"""Build libbitsmoe.so in-tree with nvcc for sm_103a (GB300).

Ten translation units, compiled in parallel: the host packer (pack.cpp,
plain C++), the CUDA kernel chain + C ABI (forward.cu), the two fused
single-token decode kernels (fused.cu, and the clustered one in fused2.cu),
the tensor-core projections (gemm.cu), the tensor-core expert factors
(expert_tc.cu), the per-unit quantiser from float spectral vectors
(quantize.cu), the per-projection bit allocation (allocate.cu) and the
importance beta from calibration tokens that the allocation weighs its losses
by (importance.cu), and the shared-basis decomposition with the calibration
Gram (decompose.cu).  The CUDA runtime is linked statically, so the library
loads on a machine without a GPU (the host-only entry points then work; the
device ones return BITSMOE_ERR_CUDA).
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libbitsmoe.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON = ["-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-lineinfo"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the BitsMoE CUDA library cannot be built")


def _run(cmd):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("build step failed:\n" + " ".join(cmd) + "\n" + r.stdout + r.stderr)
    return r.stdout + r.stderr


def sources():
    return [os.path.join(CSRC, f) for f in ("pack.cpp", "forward.cu", "fused.cu", "fused2.cu", "gemm.cu", "expert_tc.cu",
                                              "quantize.cu", "allocate.cu", "importance.cu", "decompose.cu")]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    deps = sources() + [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [
        os.path.join(HERE, "..", "include", "bitsmoe.h"), os.path.abspath(__file__)]
    return all(os.path.getmtime(d) <= t for d in deps if os.path.exists(d))


def build(force: bool = False, verbose: bool = False, extra_flags=()) -> str:
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    nv = nvcc()
    jobs = []
    for src in sources():
        obj = os.path.join(BUILD, os.path.basename(src) + ".o")
        flags = list(extra_flags) + (["-Xptxas", "-v"] if verbose and src.endswith(".cu") else [])
        jobs.append(([nv, *ARCH, *COMMON, *flags, "-I", os.path.join(HERE, "..", "include"),
                      "-c", src, "-o", obj], obj))
    with ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        logs = list(ex.map(lambda j: _run(j[0]), jobs))
    if verbose:
        for log in logs:
            sys.stdout.write(log)
    tmp = LIB + ".tmp"
    _run([nv, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *[o for _, o in jobs], "-lpthread"])
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose="-v" in sys.argv)
    print(LIB)
