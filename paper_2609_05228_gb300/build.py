"""Builds libace.so in-tree (paper_2609_05228_gb300/_lib/) with nvcc for sm_103a,
its debug variant libace_debug.so (-DACE_DEBUG_CHECKS: index guards and
canary words), and libace_offline.so (the host-only offline table tool) with g++.

Each .cu file under csrc/ is compiled in parallel, then linked into one
shared library (CUDA runtime linked statically). Run as
`python -m paper_2609_05228_gb300.build`.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIBDIR = os.path.join(PKG, "_lib")
OBJDIR = os.path.join(LIBDIR, "obj")
LIBNAME = "libace.so"
LIBPATH = os.path.join(LIBDIR, LIBNAME)

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
              "--expt-relaxed-constexpr", "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def sources() -> list[str]:
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


OFFLINE_SRC = os.path.join(PKG, "csrc_host", "ace_offline.cpp")
OFFLINE_LIB = os.path.join(LIBDIR, "libace_offline.so")


def build_offline() -> str:
    """libace_offline.so: the host-only offline GSP/RCR tool (plain C++, no CUDA)."""
    os.makedirs(LIBDIR, exist_ok=True)
    cxx = shutil.which("g++") or "g++"
    tmp = OFFLINE_LIB + ".tmp"
    cmd = [cxx, "-O3", "-std=c++17", "-fPIC", "-shared", "-pthread", "-I", INCLUDE, "-o", tmp, OFFLINE_SRC]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"g++ failed for {OFFLINE_SRC}:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, OFFLINE_LIB)
    return OFFLINE_LIB


DEBUG_LIBPATH = os.path.join(LIBDIR, "libace_debug.so")
# the debug variant: index guards in the routing, compaction, gather and
# combine kernels, canary words past every device array of a layer
DEBUG_FLAGS = ["-DACE_DEBUG_CHECKS"]


def build(verbose: bool = False, extra_flags: list[str] | None = None, debug: bool = True) -> str:
    """Compile every .cu file for both variants in parallel and link
    libace.so (and libace_debug.so unless debug=False). Returns libace.so's path."""
    cc = nvcc()
    variants = [("release", NVCC_FLAGS + (extra_flags or []), LIBPATH)]
    if debug:
        variants.append(("debug", NVCC_FLAGS + DEBUG_FLAGS + (extra_flags or []), DEBUG_LIBPATH))
    for name, _, _ in variants:
        os.makedirs(os.path.join(OBJDIR, name), exist_ok=True)

    def compile_one(job) -> str:
        src, name, flags = job
        obj = os.path.join(OBJDIR, name, os.path.basename(src)[:-3] + ".o")
        cmd = [cc, *ARCH, *flags, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src} ({name}):\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout + r.stderr, file=sys.stderr)
        return obj

    srcs = sources()
    jobs = [(src, name, flags) for name, flags, _ in variants for src in srcs]
    with ThreadPoolExecutor(max(1, min(len(jobs) + 1, os.cpu_count() or 1))) as ex:
        host = ex.submit(build_offline)
        objs = list(ex.map(compile_one, jobs))
        host.result()
    for i, (name, _, path) in enumerate(variants):
        tmp = path + ".tmp"
        cmd = [cc, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *objs[i * len(srcs):(i + 1) * len(srcs)]]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed ({name}):\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, path)
    return LIBPATH


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, extra_flags=["-Xptxas", "-v"] if "--ptxas" in sys.argv else None))
