"""Builds the CUDA library libdfs.so in-tree for sm_103a (no CMake).

Every .cu translation unit under csrc/ is compiled in parallel with nvcc, then linked
into paper_2607_06631_gb300/_lib/libdfs.so with the CUDA runtime linked statically.
Objects go to _build/ at the repository root; both folders are git-ignored.  A SHA-256
fingerprint of the sources, header, flags, compiler version and machine type is stored
beside the library, and the library is rebuilt whenever it differs.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import platform
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB_DIR = os.path.join(PKG, "_lib")
LIB = os.path.join(LIB_DIR, "libdfs.so")
STAMP = LIB + ".sha256"
BUILD = os.path.join(ROOT, "_build")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-I" + INCLUDE]
LINK = ["-shared", "-cudart", "static"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _fingerprint() -> str:
    """SHA-256 over every source the library is built from (the .cu / .cuh files and the
    public header), the compiler flags, the nvcc version and the host machine type."""
    h = hashlib.sha256()
    deps = sorted(sources() + [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cuh")])
    deps.append(os.path.join(INCLUDE, "dfs.h"))
    for d in deps:
        h.update(os.path.relpath(d, ROOT).encode())
        with open(d, "rb") as f:
            h.update(hashlib.sha256(f.read()).digest())
    h.update(" ".join(ARCH + FLAGS[:-1] + LINK).encode())
    r = subprocess.run([_nvcc(), "--version"], capture_output=True, text=True)
    h.update(r.stdout.encode())
    h.update(platform.machine().encode())
    return h.hexdigest()


def _stale(fp: str) -> bool:
    """The library is rebuilt unless it exists and the fingerprint stored beside it at its
    last build equals the current one (file times play no part)."""
    if not (os.path.exists(LIB) and os.path.exists(STAMP)):
        return True
    with open(STAMP) as f:
        return f.read().strip() != fp


def build(force: bool = False, verbose: bool = False) -> str:
    """Compiles (if needed) and returns the path of libdfs.so."""
    fp = _fingerprint()
    if not force and not _stale(fp):
        return LIB
    nvcc = _nvcc()
    os.makedirs(BUILD, exist_ok=True)
    os.makedirs(LIB_DIR, exist_ok=True)

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.basename(src)[:-3] + ".o")
        cmd = [nvcc] + ARCH + FLAGS + ["-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed on %s:\n%s%s" % (src, r.stdout, r.stderr))
        if verbose:
            print(" ".join(cmd))
        return obj

    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        objs = list(ex.map(compile_one, sources()))
    tmp = LIB + ".tmp"
    cmd = [nvcc] + ARCH + LINK + ["-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
    os.replace(tmp, LIB)
    with open(STAMP, "w") as f:
        f.write(fp + "\n")
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
