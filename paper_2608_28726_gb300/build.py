"""Build step of libprorouter.so (sm_103a only, compiled in-tree).

    python -m paper_2608_28726_gb300.build          # build if sources changed
    python -m paper_2608_28726_gb300.build --force  # rebuild

nvcc cross-compiles without a GPU.  The translation units under csrc/ are
compiled in parallel and linked into one shared library; it links the CUDA
runtime statically, so it depends only on the driver at run time.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(OUT_DIR, "libprorouter.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libprorouter.so")


def sources() -> list[str]:
    files = [os.path.join(CSRC, f) for f in sorted(os.listdir(CSRC))]
    return [f for f in files if f.endswith((".cu", ".cuh", ".h"))] + [
        os.path.join(INCLUDE, "pro_router.h")]


def stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in sources())


def units() -> list[str]:
    """Translation units of the library (compiled in parallel, then linked)."""
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and not stale():
        return LIB
    os.makedirs(OUT_DIR, exist_ok=True)
    tag = ".tmp%d" % os.getpid()
    flags = [*ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE]
    if verbose:
        flags.insert(0, "-Xptxas=-v")
    objs, procs = [], []
    for src in units():
        obj = os.path.join(OUT_DIR, os.path.basename(src)[:-3] + tag + ".o")
        objs.append(obj)
        procs.append((src, subprocess.Popen([nvcc(), *flags, "-c", src, "-o", obj])))
    failed = [src for src, p in procs if p.wait() != 0]
    if failed:
        for obj in objs:
            if os.path.exists(obj):
                os.remove(obj)
        raise subprocess.CalledProcessError(1, "nvcc -c " + " ".join(failed))
    tmp = LIB + tag
    try:
        subprocess.check_call([nvcc(), *ARCH, "-shared", *objs, "-o", tmp])
    finally:
        for obj in objs:
            os.remove(obj)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
