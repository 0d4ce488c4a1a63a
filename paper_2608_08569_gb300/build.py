"""Builds ``libvoxzip.so`` (the C-ABI CUDA library) in-tree for sm_103a with nvcc.

Each ``csrc/*.cu`` file compiles to an object in ``_build/`` in parallel, then nvcc links the
shared library next to this file. ``python -m paper_2608_08569_gb300.build`` runs it.

``--checked`` builds ``libvoxzip_checked.so`` instead, with ``-DVOXZIP_CHECKED``: its kernels
range-check the indices of their global accesses, skip an access that is out of range and set
``VOXZIP_DEV_BOUNDS`` in the status word. Setting ``VOXZIP_CHECKED=1`` in the environment makes
the binding load that library.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG_DIR)
CSRC = os.path.join(PKG_DIR, "csrc")
BUILD_DIR = os.path.join(ROOT, "_build")
LIB_PATH = os.path.join(PKG_DIR, "libvoxzip.so")
CHECKED_LIB_PATH = os.path.join(PKG_DIR, "libvoxzip_checked.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "-cudart", "shared",
              "--expt-relaxed-constexpr", "-Xptxas", "-v", "-I" + os.path.join(ROOT, "include")]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libvoxzip.so")


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + sorted(glob.glob(os.path.join(CSRC, "*.cuh"))) + [
        os.path.join(ROOT, "include", "voxzip.h")]


def up_to_date(checked: bool = False) -> bool:
    lib_path = CHECKED_LIB_PATH if checked else LIB_PATH
    if not os.path.exists(lib_path):
        return False
    t = os.path.getmtime(lib_path)
    return all(os.path.getmtime(p) <= t for p in _deps())


def build_library(force: bool = False, verbose: bool = False, checked: bool = False) -> str:
    """Compile and link ``libvoxzip.so`` (``libvoxzip_checked.so`` with `checked`); returns its
    path. Skips work when up to date."""
    lib_path = CHECKED_LIB_PATH if checked else LIB_PATH
    if not force and up_to_date(checked):
        return lib_path
    nvcc = _nvcc()
    build_dir = os.path.join(BUILD_DIR, "checked") if checked else BUILD_DIR
    os.makedirs(build_dir, exist_ok=True)
    srcs = _sources()
    flags = NVCC_FLAGS + (["-DVOXZIP_CHECKED"] if checked else [])

    def compile_one(src):
        obj = os.path.join(build_dir, os.path.basename(src)[:-3] + ".o")
        cmd = [nvcc, *ARCH, *flags, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        with open(obj + ".ptxas.txt", "w") as f:
            f.write(r.stderr)
        return obj

    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(srcs), os.cpu_count() or 1))) as ex:
        objs = list(ex.map(compile_one, srcs))
    tmp = lib_path + f".tmp{os.getpid()}"
    cmd = [nvcc, *ARCH, "-shared", "-cudart", "shared", "-Xlinker", "-rpath,/usr/local/cuda/lib64", "-o", tmp,
           *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib_path)
    if verbose:
        for o in objs:
            with open(o + ".ptxas.txt") as f:
                sys.stdout.write(f.read())
    return lib_path


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose="-v" in sys.argv, checked="--checked" in sys.argv))
