"""Build libmone.so in-tree with nvcc for sm_103a (no cmake, no torch extension).

Each translation unit is compiled in parallel; the shared library links the
CUDA runtime statically, so it loads on a machine without a GPU driver (the
C-ABI symbol checks run there) and needs nothing but the driver on a GPU machine.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libmone.so")
SOURCES = ["mone_api.cu", "ttl_prepass.cu", "ttl_simt.cu", "ttl_tc.cu", "attention.cu", "swiglu_tc.cu", "host_stage.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _flags(extra=()):
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include"),
                   "-I", CSRC, *extra]


def _digest(paths, extra=()) -> str:
    """sha256 over file contents and strings: build outputs are reused only when this matches
    the stamp written beside them (content, not modification times, which need not be
    comparable between the machine that edited the sources and the one that builds)."""
    h = hashlib.sha256()
    for p in sorted(paths):
        h.update(p.encode())
        with open(p, "rb") as f:
            h.update(f.read())
    for e in extra:
        h.update(str(e).encode())
    return h.hexdigest()


def _fresh(target: str, digest: str) -> bool:
    try:
        with open(target + ".sha") as f:
            return os.path.exists(target) and f.read().strip() == digest
    except OSError:
        return False


def _stamp(target: str, digest: str) -> None:
    with open(target + ".sha", "w") as f:
        f.write(digest)


def build(verbose: bool = False, force: bool = False, ptxas_info: bool = False, debug: bool = False) -> str:
    """Compile every translation unit and link libmone.so.  debug=True builds the MONE_DEBUG
    variant instead (device-side index checks on, -lineinfo as always) into libmone_debug.so,
    with its objects apart; load it with MONE_LIB=<path>."""
    BUILD = os.path.join(PKG, "_build_debug" if debug else "_build")
    LIB = os.path.join(PKG, "libmone_debug.so" if debug else "libmone.so")
    os.makedirs(BUILD, exist_ok=True)
    headers = [os.path.join(CSRC, h) for h in os.listdir(CSRC) if h.endswith((".h", ".cuh"))]
    headers.append(os.path.join(ROOT, "include", "mone.h"))
    cc = nvcc()
    extra = (["-Xptxas", "-v"] if ptxas_info else []) + (["-DMONE_DEBUG"] if debug else [])

    machine = os.uname().machine

    def compile_one(src):
        s = os.path.join(CSRC, src)
        o = os.path.join(BUILD, src.replace(".cu", ".o"))
        cmd = [cc, *_flags(extra), "-c", s, "-o", o]
        digest = _digest([s, *headers], [machine, *cmd])
        if not force and not ptxas_info and _fresh(o, digest):
            return o, "", digest
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        _stamp(o, digest)
        return o, r.stderr, digest

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    objs = [o for o, _, _ in results]
    if verbose or ptxas_info:
        for _, log, _ in results:
            if log:
                sys.stderr.write(log)
    cmd = [cc, *ARCH, "-shared", "-o", LIB + ".tmp", *objs, "-cudart", "static", "-Xcompiler", "-fPIC"]
    digest = _digest([], [machine, *cmd, *[d for _, _, d in results]])
    if force or ptxas_info or not _fresh(LIB, digest):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(LIB + ".tmp", LIB)
        _stamp(LIB, digest)
    return LIB


if __name__ == "__main__":
    print(build(verbose=True, force="--force" in sys.argv, ptxas_info="--ptxas" in sys.argv,
                debug="--debug" in sys.argv))
