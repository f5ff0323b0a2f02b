"""Builds libevisel.so in-tree for sm_103a (nvcc only, no cmake).

Each translation unit is compiled in parallel; the shared library links the
CUDA runtime statically and reaches the driver API through the runtime's
entry-point query, so it needs nothing beyond the NVIDIA driver at run time.

The library carries a build id: a SHA-256 over its sources and headers, this
script, the compiler flags, the nvcc version and the host machine type,
compiled in as a string and returned by evisel_build_id(). build() rebuilds
whenever the library on disk does not hold the id of the current tree, so a
stale or foreign libevisel.so is never the one that runs.
"""
from __future__ import annotations

import hashlib
import os
import platform
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libevisel.so")

SOURCES = ["probe_attn.cu", "attn_combine.cu", "evidence.cu", "evisel_capi.cpp", "evisel_noalloc.cu", "evisel_selftest.cu", "intra_frame.cu",
           "cross_frame.cu", "text_evidence.cu", "topp_mask.cu",
           "coarse_evidence.cu"]
HEADERS = ["evisel_internal.h", "evisel_plan.h", "sm103_ptx.cuh"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
         "--expt-relaxed-constexpr", "-I" + INCLUDE, "-I" + CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


ID_PREFIX = b"evisel-build-id:"


def build_id() -> str:
    """SHA-256 (first 24 hex digits) of everything that determines the binary."""
    h = hashlib.sha256()
    for f in [os.path.join(CSRC, f) for f in SOURCES + HEADERS] + [os.path.join(INCLUDE, "evisel.h"), __file__]:
        h.update(os.path.basename(f).encode() + b"\0")
        with open(f, "rb") as fh:
            h.update(fh.read())
    h.update(" ".join(ARCH + FLAGS).replace(INCLUDE, "<include>").replace(CSRC, "<csrc>").encode())
    try:
        ver = subprocess.run([nvcc(), "--version"], capture_output=True, text=True).stdout
    except (OSError, RuntimeError):
        ver = "nvcc-unavailable"
    h.update(ver.encode())
    h.update(platform.machine().encode())
    return h.hexdigest()[:24]


def library_id(path: str = LIB) -> str | None:
    """The build id compiled into the library at ``path`` (None if absent)."""
    if not os.path.exists(path):
        return None
    with open(path, "rb") as fh:
        data = fh.read()
    i = data.find(ID_PREFIX)
    if i < 0:
        return None
    return data[i + len(ID_PREFIX):i + len(ID_PREFIX) + 24].decode("ascii", "replace")


def build(force: bool = False, verbose: bool = False) -> str:
    """Compiles the library unless it already holds the current build id; returns its path."""
    want = build_id()
    if not force and library_id() == want:
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.splitext(src)[0] + ".o")
        extra = ["-Xptxas", "-v"] if verbose and src.endswith(".cu") else []
        cmd = [cc, *ARCH, *FLAGS, *extra, f"-DEVISEL_BUILD_ID=\"{want}\"", "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"compile failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose:
        for _, log in results:
            sys.stderr.write(log)
    tmp = LIB + ".tmp"
    cmd = [cc, *ARCH, "-shared", "-o", tmp, *[o for o, _ in results]]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    if library_id() != want:
        raise RuntimeError("the built library does not carry the expected build id")
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv), build_id())
