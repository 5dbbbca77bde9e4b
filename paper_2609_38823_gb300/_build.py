"""Build libdecomoe.so in-tree with nvcc for sm_103a.

Each CUDA translation unit compiles in parallel (one -gencode), the plain-C
prefix selection with gcc, and nvcc links the shared library next to this file.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
ROOT = os.path.dirname(HERE)
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(HERE, "libdecomoe.so")

CU_SOURCES = ["api.cu", "route.cu", "dispatch.cu", "expert_gemm.cu", "combine_compact.cu", "calib_gate.cu", "layer.cu", "decode_layer.cu", "attention.cu"]
C_SOURCES = ["prefix.c"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc_path() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found")
    return cand


def _run(cmd):
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError("command failed:\n" + " ".join(cmd) + "\n" + r.stdout)
    return r.stdout


def build(verbose: bool = False, ptxas_info: bool = False, force: bool = False) -> str:
    os.makedirs(BUILD, exist_ok=True)
    nvcc = nvcc_path()
    srcs = [os.path.join(CSRC, s) for s in CU_SOURCES + C_SOURCES]
    hdrs = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cuh")]
    hdrs.append(os.path.join(ROOT, "include", "decomoe.h"))
    if not force and os.path.exists(LIB):
        lib_t = os.path.getmtime(LIB)
        if all(os.path.getmtime(p) < lib_t for p in srcs + hdrs + [__file__]):
            return LIB
    common = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-fvisibility=hidden",
              "--expt-relaxed-constexpr", "-I" + os.path.join(ROOT, "include")]
    if ptxas_info:
        common += ["-Xptxas", "-v"]
    jobs = []
    for s in CU_SOURCES:
        obj = os.path.join(BUILD, s.replace(".cu", ".o"))
        jobs.append(([nvcc, *ARCH, *common, "-c", os.path.join(CSRC, s), "-o", obj], obj))
    for s in C_SOURCES:
        obj = os.path.join(BUILD, s.replace(".c", ".c.o"))
        cc = shutil.which("gcc") or "cc"
        jobs.append(([cc, "-O2", "-std=c11", "-fPIC", "-fvisibility=hidden", "-Wall",
                      "-I" + os.path.join(ROOT, "include"), "-c", os.path.join(CSRC, s), "-o", obj], obj))
    outs = []
    with cf.ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 4)) as ex:
        for out in ex.map(lambda j: _run(j[0]), jobs):
            outs.append(out)
    if verbose or ptxas_info:
        for o in outs:
            if o.strip():
                sys.stdout.write(o)
    tmp = LIB + ".tmp"
    _run([nvcc, *ARCH, "-shared", "-o", tmp, *[j[1] for j in jobs], "-lcudart"])
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(verbose=True, ptxas_info="-v" in sys.argv, force="-f" in sys.argv)
    print(LIB)
