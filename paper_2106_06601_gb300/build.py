"""Builds the CUDA library in-tree: paper_2106_06601_gb300/_build/libcosta_gb300.so.

Kernels are compiled by nvcc for sm_103a only; host C++ by g++; the
translation units compile in parallel and nvcc links them with the static
CUDA runtime.  No cmake, no torch extension machinery.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(BUILD, "libcosta_gb300.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home and os.path.exists(os.path.join(home, "bin", "nvcc")):
        return home
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return "/usr/local/cuda"


def sources():
    cu = sorted(f for f in os.listdir(CSRC) if f.endswith(".cu"))
    cpp = sorted(f for f in os.listdir(CSRC) if f.endswith(".cpp"))
    hdr = sorted(f for f in os.listdir(CSRC) if f.endswith((".h", ".cuh")))
    return cu, cpp, hdr


def _stale(objs_and_srcs) -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in objs_and_srcs)


def build(force: bool = False, verbose: bool = False, extra_nvcc=(), defines=()) -> str:
    """Compiles every translation unit and links the library.  `defines`
    (-DNAME=VALUE) go to both compilers (tuning overrides)."""
    os.makedirs(BUILD, exist_ok=True)
    cu, cpp, hdr = sources()
    deps = [os.path.join(CSRC, f) for f in cu + cpp + hdr] + [os.path.join(INCLUDE, "costa_gb300.h"),
                                                              os.path.abspath(__file__)]
    if not force and not _stale(deps):
        return LIB
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    incs = ["-I", INCLUDE, "-I", CSRC]
    jobs, objs = [], []
    for f in cu:
        obj = os.path.join(BUILD, f + ".o")
        cmd = [nvcc, *ARCH, "-lineinfo", "-O3", "-std=c++17", "-Xcompiler", "-fPIC",
               "-Xptxas", "-v" if verbose else "-O3", *extra_nvcc, *defines, *incs,
               "-c", os.path.join(CSRC, f), "-o", obj]
        jobs.append((cmd, f))
        objs.append(obj)
    for f in cpp:
        obj = os.path.join(BUILD, f + ".o")
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-Wall", "-Wextra", "-Wno-unused-parameter",
               *defines, *incs, "-I", os.path.join(cuda, "include"), "-c", os.path.join(CSRC, f), "-o", obj]
        jobs.append((cmd, f))
        objs.append(obj)
    procs = [(subprocess.Popen(c, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True), f)
             for c, f in jobs]
    failed = []
    for p, f in procs:
        out, _ = p.communicate()
        if verbose or p.returncode != 0:
            sys.stderr.write(f"--- {f}\n{out}")
        if p.returncode != 0:
            failed.append(f)
    if failed:
        raise RuntimeError(f"compilation failed: {failed}")
    tmp = LIB + f".tmp{os.getpid()}"
    link = [nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"]
    r = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        sys.stderr.write(r.stdout)
        raise RuntimeError("link failed")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
