"""Builds libsq.so (CUDA, sm_103a) and libsq_host.so (host logic only, for
CPU tests) in-tree under paper_2602_22603_gb300/_build/.

nvcc compiles each translation unit in parallel; the objects are linked
with the static CUDA runtime into one shared library with a plain C ABI.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT = os.path.join(PKG, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-use_fast_math", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-fvisibility=hidden", "-I" + INCLUDE]

LIBSQ_SOURCES = [
    "kernels/decode.cu",
    "kernels/kv.cu",
    "kernels/noalloc_scratch.cu",
    "kernels/prefill.cu",
    "kernels/probe.cu",
    "host/core.cpp",
    "api/sq_api.cpp",
]
HOST_SOURCES = ["host/core.cpp", "api/host_test_api.cpp"]

LIBSQ = os.path.join(OUT, "libsq.so")
LIBSQ_HOST = os.path.join(OUT, "libsq_host.so")


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _all_sources():
    out = []
    for d, _, files in os.walk(CSRC):
        for f in files:
            if f.endswith((".cu", ".cuh", ".cpp", ".hpp", ".h")):
                out.append(os.path.join(d, f))
    out.append(os.path.join(INCLUDE, "sq.h"))
    return out


def _stale(target: str) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(s) > t for s in _all_sources())


def _run(cmd):
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError("build step failed:\n" + " ".join(cmd) + "\n" + r.stdout)
    return r.stdout


def build_libsq(force: bool = False, verbose: bool = False, extra=()) -> str:
    if not force and not _stale(LIBSQ):
        return LIBSQ
    os.makedirs(OUT, exist_ok=True)
    nvcc = _nvcc()
    objs = []
    cmds = []
    for src in LIBSQ_SOURCES:
        obj = os.path.join(OUT, src.replace("/", "_") + ".o")
        objs.append(obj)
        cmds.append([nvcc, *ARCH, *NVCC_FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj])
    with cf.ThreadPoolExecutor(max_workers=len(cmds)) as ex:
        logs = list(ex.map(_run, cmds))
    if verbose:
        for log in logs:
            if log.strip():
                print(log)
    tmp = LIBSQ + f".tmp{os.getpid()}"
    _run([nvcc, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *objs])
    os.replace(tmp, LIBSQ)
    return LIBSQ


def build_host_lib(force: bool = False) -> str:
    if not force and not _stale(LIBSQ_HOST):
        return LIBSQ_HOST
    os.makedirs(OUT, exist_ok=True)
    tmp = LIBSQ_HOST + f".tmp{os.getpid()}"
    _run(["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-o", tmp,
          *[os.path.join(CSRC, s) for s in HOST_SOURCES]])
    os.replace(tmp, LIBSQ_HOST)
    return LIBSQ_HOST


def build_all(force: bool = False, verbose: bool = False) -> None:
    with cf.ThreadPoolExecutor(max_workers=2) as ex:
        a = ex.submit(build_libsq, force, verbose)
        b = ex.submit(build_host_lib, force)
        a.result()
        b.result()


if __name__ == "__main__":
    build_all(force="--force" in sys.argv, verbose="-v" in sys.argv)
    print(LIBSQ)
