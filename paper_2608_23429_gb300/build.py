"""Build libchebboost.so in-tree for sm_103a (nvcc, no cmake).

Each CUDA translation unit is compiled in parallel, then linked against the
shared CUDA runtime so that the library and PyTorch share one runtime (and
stream handles pass between them unchanged).

A build is reused only when its stamp matches: a SHA-256 over every source and
header, the compiler flags, the nvcc version and the host machine type, written
into the build directory after a successful link. Any other state (a library
or object files copied from another machine, sources edited since, another
toolkit) recompiles everything. Usage:
``python -m paper_2608_23429_gb300.build [--force] [-v]``.
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
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libchebboost.so")
STAMP = os.path.join(BUILD, "stamp.sha256")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CFLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2"]
SOURCES = ["extrapolate.cu", "extrapolate_gated.cu", "extrapolate_bulk.cu", "extrapolate_bulk_gated.cu",
           "push.cu", "epilogue.cu", "static_status.cu", "plan.cpp"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libchebboost")


def _cuda_lib_dir(nvcc: str) -> str:
    return os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(nvcc))), "lib64")


def _inputs() -> list[str]:
    files = [os.path.join(CSRC, f) for f in sorted(os.listdir(CSRC)) if f.endswith((".cu", ".cpp", ".h", ".cuh"))]
    files.append(os.path.join(INCLUDE, "chebboost.h"))
    return files


def source_hash(nvcc: str) -> str:
    """Stamp of one build: sources, headers, flags, toolkit and machine."""
    h = hashlib.sha256()
    for f in _inputs():
        h.update(os.path.relpath(f, os.path.dirname(HERE)).encode())
        with open(f, "rb") as fh:
            h.update(hashlib.sha256(fh.read()).digest())
    ver = subprocess.run([nvcc, "--version"], capture_output=True, text=True).stdout
    h.update(" ".join(ARCH + CFLAGS + SOURCES).encode())
    h.update(ver.encode())
    h.update(platform.machine().encode())
    return h.hexdigest()


def _current(stamp: str) -> bool:
    if not (os.path.exists(LIB) and os.path.exists(STAMP)):
        return False
    with open(STAMP) as fh:
        return fh.read().strip() == stamp


def build(force: bool = False, verbose: bool = False) -> str:
    nvcc = _nvcc()
    stamp = source_hash(nvcc)
    if not force and _current(stamp):
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    if os.path.exists(STAMP):
        os.remove(STAMP)
    objs, jobs = [], []
    for src in SOURCES:
        s = os.path.join(CSRC, src)
        o = os.path.join(BUILD, src + ".o")
        objs.append(o)
        cmd = [nvcc, *ARCH, *CFLAGS, f"-I{INCLUDE}", "-c", s, "-o", o]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        jobs.append(cmd)

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        return cmd, r

    with ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        for cmd, r in ex.map(run, jobs):
            if verbose and r.stderr:
                sys.stderr.write(r.stderr)
            if r.returncode != 0:
                raise RuntimeError(f"build failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [nvcc, *ARCH, "-shared", "-cudart", "shared", "-o", tmp, *objs,
           "-Xlinker", f"-rpath,{_cuda_lib_dir(nvcc)}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(STAMP, "w") as fh:
        fh.write(stamp + "\n")
    print(f"libchebboost: compiled {len(SOURCES)} units for {platform.machine()} ({stamp[:12]})", file=sys.stderr)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose="-v" in sys.argv)
    print(LIB)
