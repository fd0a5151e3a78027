"""Build libtreepo.so in-tree with nvcc for sm_103a (GB300).

Run ``python -m paper_2508_17445_gb300.build`` or call ``build()``. Sources
compile in parallel; the host C++ goes through nvcc's host compiler with
portable flags only (the library is built on x86_64 and on aarch64).

``build(checked=True)`` builds the bounds-checked variant,
libtreepo_checked.so: the same sources with TP_BOUNDS_CHECK defined, so every
kernel checks the schedule indices it uses before each access and reports a
failed check through tp_sync instead of touching memory out of bounds. The
binding loads it instead of libtreepo.so when TREEPO_BOUNDS_CHECK=1 is set.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
ROOT = os.path.dirname(HERE)
LIB = os.path.join(HERE, "libtreepo.so")
LIB_CHECKED = os.path.join(HERE, "libtreepo_checked.so")
BUILD_DIR = os.path.join(HERE, "_build")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
SOURCES = ["kernels.cu", "forest.cpp", "capi.cpp", "rollout.cpp"]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libtreepo")


def _stale(lib: str) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(ROOT, "include", "treepo.h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False, checked: bool = False) -> str:
    lib = LIB_CHECKED if checked else LIB
    if not force and not _stale(lib):
        return lib
    nvcc = _nvcc()
    build_dir = BUILD_DIR + ("_checked" if checked else "")
    os.makedirs(build_dir, exist_ok=True)
    common = ["-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include")]
    if checked:
        common.append("-DTP_BOUNDS_CHECK")

    def compile_one(src: str) -> str:
        obj = os.path.join(build_dir, src + ".o")
        cmd = [nvcc, *common, "-c", os.path.join(CSRC, src), "-o", obj]
        if src.endswith(".cu"):
            cmd[1:1] = [*ARCH, "-lineinfo", "-Xptxas", "-v" if verbose else "-O3"]
        else:
            # no fused multiply-add contraction: host decisions that compare
            # doubles (branch splits) must round the same on every machine
            cmd[1:1] = ["-x", "c++", "-Xcompiler", "-ffp-contract=off"]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"compiling {src} failed:\n{' '.join(cmd)}\n{res.stdout}\n{res.stderr}")
        if verbose and res.stderr:
            sys.stderr.write(res.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    tmp = lib + f".{os.getpid()}.tmp"
    cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"linking {os.path.basename(lib)} failed:\n{' '.join(cmd)}\n{res.stdout}\n{res.stderr}")
    os.replace(tmp, lib)
    return lib


def build_all(force: bool = False) -> None:
    """Both variants, in parallel (each compiles its sources in parallel)."""
    with ThreadPoolExecutor(max_workers=2) as ex:
        list(ex.map(lambda c: build(force=force, checked=c), (False, True)))


if __name__ == "__main__":
    if "--checked" in sys.argv:
        print(build(force="--force" in sys.argv, verbose="-v" in sys.argv, checked=True))
    else:
        print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
