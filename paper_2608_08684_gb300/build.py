"""In-tree build of libripple.so (CUDA kernels for sm_103a + the host C allocator).

Each translation unit is compiled in parallel with nvcc (CUDA) or gcc (C), then
linked with nvcc into paper_2608_08684_gb300/libripple.so. The build is skipped
when the library is newer than every source and header.

build_library(checked=True) builds libripple_checked.so from the same sources
with RIPPLE_CHECKED defined: every guarded global access in the kernels tests
its offset against its buffer's extent and reports RIPPLE_EBOUNDS in the
call's status word instead of going out of bounds (the bounds-check build that
stands in for a memory checker; the binding loads it when RIPPLE_CHECKED=1 is
set in the environment).
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libripple.so")
BUILD_CHECKED = os.path.join(PKG, "_build_checked")
LIB_CHECKED = os.path.join(PKG, "libripple_checked.so")

NVCC = os.environ.get("NVCC", "nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                     "-Xcompiler", "-ffp-contract=off", "-I", INCLUDE, "-I", CSRC]
CC_FLAGS = ["-O2", "-std=c99", "-fPIC", "-ffp-contract=off", "-Wall", "-I", INCLUDE]


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu"))) + sorted(glob.glob(os.path.join(CSRC, "*.c")))


def _deps():
    return _sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))


def _stale(lib: str) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    return any(os.path.getmtime(p) > t for p in _deps())


def _compile(src: str, extra: list, build_dir: str) -> str:
    obj = os.path.join(build_dir, os.path.basename(src) + ".o")
    if src.endswith(".cu"):
        cmd = [NVCC] + NVCC_FLAGS + extra + ["-c", src, "-o", obj]
    else:
        cmd = [os.environ.get("CC", "gcc")] + CC_FLAGS + ["-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"compile failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    return obj


def build_library(force: bool = False, verbose: bool = False, extra_nvcc=(),
                  checked: bool = False) -> str:
    """Build libripple.so (libripple_checked.so with checked=True) if it is
    missing or older than its sources; return its path."""
    lib, build_dir = (LIB_CHECKED, BUILD_CHECKED) if checked else (LIB, BUILD)
    extra = list(extra_nvcc) + (["-DRIPPLE_CHECKED"] if checked else [])
    if not force and not _stale(lib):
        return lib
    os.makedirs(build_dir, exist_ok=True)
    srcs = _sources()
    with cf.ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra, build_dir), srcs))
    tmp = lib + ".tmp"
    cmd = [NVCC] + ARCH + ["-shared", "-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    if verbose:
        print(f"built {lib}", file=sys.stderr)
    return lib


if __name__ == "__main__":
    build_library(force="--force" in sys.argv, verbose=True, checked="--checked" in sys.argv)
