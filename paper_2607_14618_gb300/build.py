"""In-tree build of ``libpolyq.so`` (host C++ + sm_103a CUDA kernels).

Compiles every translation unit under ``csrc/`` in parallel and links one
shared library next to this file.  Host code is built with
``-ffp-contract=off`` so that packing arithmetic is plain IEEE double in
program order on any host.
"""
from __future__ import annotations

import glob
import os
import platform
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libpolyq.so")
STAMP = os.path.join(BUILD, "stamp.txt")
# The debug build (-DPOLYQ_DEBUG, a test aid): the same sources, whose GEMV
# and GEMM kernels also write the codes and weights they decode.
BUILD_DEBUG = os.path.join(HERE, "_build_debug")
LIB_DEBUG = os.path.join(HERE, "libpolyq_debug.so")
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def _cuda_home():
    for c in (os.environ.get("CUDA_HOME"), "/usr/local/cuda"):
        if c and os.path.exists(os.path.join(c, "bin", "nvcc")):
            return c
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(nvcc))
    raise RuntimeError("nvcc not found: set CUDA_HOME")


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cpp")) + glob.glob(os.path.join(CSRC, "*.cu")))


def _headers():
    return sorted(glob.glob(os.path.join(CSRC, "*.h")) + glob.glob(os.path.join(CSRC, "*.cuh"))
                  + glob.glob(os.path.join(INCLUDE, "*.h")))


def _stamp_text():
    return f"{platform.machine()} {sys.version_info[:2]}"


def _up_to_date(lib, build):
    stamp = os.path.join(build, "stamp.txt")
    if not os.path.exists(lib) or not os.path.exists(stamp):
        return False
    with open(stamp) as f:
        if f.read().strip() != _stamp_text():
            return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _sources() + _headers() + [__file__])


def build_library(force: bool = False, verbose: bool = False, debug: bool = False) -> str:
    """Build (if stale) and return the path of libpolyq.so (or, with
    ``debug``, of the test aid libpolyq_debug.so)."""
    lib, build = (LIB_DEBUG, BUILD_DEBUG) if debug else (LIB, BUILD)
    if not force and _up_to_date(lib, build):
        return lib
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    os.makedirs(build, exist_ok=True)
    inc = ["-I", INCLUDE, "-I", CSRC, "-I", os.path.join(cuda, "include")]
    defs = ["-DPOLYQ_DEBUG"] if debug else []
    jobs = []
    objs = []
    for src in _sources():
        obj = os.path.join(build, os.path.basename(src) + ".o")
        objs.append(obj)
        if src.endswith(".cu"):
            cmd = [nvcc, "-O3", "-std=c++17", ARCH, "-lineinfo", "--expt-relaxed-constexpr",
                   "-Xcompiler", "-fPIC,-ffp-contract=off", "-Xptxas", "-warn-spills",
                   *defs, *inc, "-c", src, "-o", obj]
        else:
            cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-ffp-contract=off", "-Wall",
                   *defs, *inc, "-c", src, "-o", obj]
        jobs.append((cmd, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)))
    failed = []
    for cmd, p in jobs:
        out, _ = p.communicate()
        text = out.decode(errors="replace")
        if p.returncode != 0:
            failed.append(" ".join(cmd) + "\n" + text)
        elif verbose and text.strip():
            print(text)
    if failed:
        raise RuntimeError("libpolyq build failed:\n" + "\n".join(failed))
    tmp = lib + ".tmp"
    link = [nvcc, "-shared", ARCH, "-cudart=shared", "-o", tmp, *objs,
            "-Xlinker", "-rpath," + os.path.join(cuda, "lib64"), "-lpthread"]
    p = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)
    if p.returncode != 0:
        raise RuntimeError("libpolyq link failed:\n" + " ".join(link) + "\n"
                           + p.stdout.decode(errors="replace"))
    os.replace(tmp, lib)
    with open(os.path.join(build, "stamp.txt"), "w") as f:
        f.write(_stamp_text())
    return lib


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose=True))
