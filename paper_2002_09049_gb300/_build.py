"""Builds libmpq.so (the C-ABI library) in-tree from csrc/*.cu with nvcc for sm_103a.

Translation units compile in parallel, then link into one shared library with the CUDA runtime
linked statically.  Run ``python -m paper_2002_09049_gb300._build`` or call ``build()``.
``build(checked=True)`` (``--checked``) builds the checked library, libmpq_checked.so: the same
sources with -DMPQ_CHECK_BOUNDS, whose kernels count and skip out-of-range accesses.
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import sys
import threading
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libmpq.so")
CHECKED_LIB = os.path.join(PKG, "libmpq_checked.so")
ROOT = os.path.dirname(PKG)
INCLUDE = os.path.join(ROOT, "include")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "-I", INCLUDE,
              "-Xptxas", "-warn-spills"]
_lock = threading.Lock()


def nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libmpq.so")
    return cand


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + [os.path.join(INCLUDE, "mpq.h")]


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _deps())


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False,
          checked: bool = False) -> str:
    """Compile csrc/*.cu -> libmpq.so, or with checked=True -> libmpq_checked.so (skipped when
    up to date).  Returns the library path."""
    lib = CHECKED_LIB if checked else LIB
    obj_dir = os.path.join(BUILD, "checked") if checked else BUILD
    with _lock:
        if not force and up_to_date(lib):
            return lib
        os.makedirs(obj_dir, exist_ok=True)
        exe = nvcc()
        extra = ["-Xptxas", "-v"] if ptxas_info else []
        if checked:
            extra += ["-DMPQ_CHECK_BOUNDS"]

        def compile_one(src):
            obj = os.path.join(obj_dir, os.path.basename(src)[:-3] + ".o")
            cmd = [exe, *ARCH, *NVCC_FLAGS, *extra, "-c", src, "-o", obj]
            res = subprocess.run(cmd, capture_output=True, text=True)
            if res.returncode != 0:
                raise RuntimeError(f"nvcc failed on {src}:\n{res.stdout}\n{res.stderr}")
            if verbose or ptxas_info:
                sys.stderr.write(res.stdout + res.stderr)
            return obj

        with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 4)) as ex:
            objs = list(ex.map(compile_one, _sources()))
        tmp = lib + f".{os.getpid()}.tmp"
        cmd = [exe, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *objs]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"link failed:\n{res.stdout}\n{res.stderr}")
        os.replace(tmp, lib)
        return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True, ptxas_info="--ptxas" in sys.argv,
                checked="--checked" in sys.argv))
