"""Builds libblr.so (the C-ABI BD-LRU scan library) in-tree with nvcc for sm_103a.

    python -m paper_2406_12580_gb300.build [--verbose]
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
import tempfile

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIBRARY = os.path.join(PKG, "libblr.so")
SOURCES = [os.path.join(CSRC, "blr_api.cu")]
DEPENDS = SOURCES + [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))] + [
    os.path.join(INCLUDE, "blr.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc_path() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def nvcc_flags(verbose: bool = False) -> list:
    cuda_lib = os.path.join(os.path.dirname(os.path.dirname(nvcc_path())), "lib64")
    flags = [*ARCH, "-O3", "-lineinfo", "-std=c++17", "-shared", "-Xcompiler", "-fPIC",
             "-Xcompiler", "-fvisibility=hidden", "-cudart", "shared", "-I", INCLUDE, "-I", CSRC,
             "-Xlinker", f"-rpath,{cuda_lib}"]
    if verbose:
        flags += ["-Xptxas", "-v"]
    return flags


def stale() -> bool:
    if not os.path.exists(LIBRARY):
        return True
    t = os.path.getmtime(LIBRARY)
    return any(os.path.getmtime(f) > t for f in DEPENDS)


def build(verbose: bool = False, force: bool = True) -> str:
    """Compile the library (atomically replacing any previous build)."""
    if not force and not stale():
        return LIBRARY
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=PKG)
    os.close(fd)
    try:
        cmd = [nvcc_path(), *nvcc_flags(verbose), *SOURCES, "-o", tmp]
        res = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
        if res.returncode != 0:
            raise RuntimeError("nvcc failed:\n" + res.stdout)
        if verbose:
            sys.stdout.write(res.stdout)
        os.replace(tmp, LIBRARY)
    finally:
        if os.path.exists(tmp):
            os.unlink(tmp)
    return LIBRARY


if __name__ == "__main__":
    build(verbose="--verbose" in sys.argv)
    print(LIBRARY)
