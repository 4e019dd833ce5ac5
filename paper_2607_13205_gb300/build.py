"""Builds librolekv.so (the sm_103a kernels and the C ABI) in-tree with nvcc.

Each translation unit is compiled in parallel; the shared object is written
next to this file, where the Python binding loads it.  The checked build
(-DROLEKV_CHECKED: every computed global access checked against its buffer's
extent, a miss reported in the status word and skipped) is a second library,
librolekv_checked.so, from the same sources.
"""

from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG_DIR)
CSRC = os.path.join(PKG_DIR, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(ROOT, "_build")
LIB_PATH = os.path.join(PKG_DIR, "librolekv.so")
CHECKED_BUILD_DIR = os.path.join(ROOT, "_build", "checked")
CHECKED_LIB_PATH = os.path.join(PKG_DIR, "librolekv_checked.so")

SOURCES = ["rolekv_api.cu", "attn_score.cu", "select.cu", "compact.cu", "quest.cu", "decode.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc_path() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found; the CUDA toolkit is required to build librolekv")
    return cand


def _compile(nvcc: str, src: str, extra: list[str], build_dir: str = BUILD_DIR) -> str:
    obj = os.path.join(build_dir, os.path.splitext(src)[0] + ".o")
    cmd = [nvcc, *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
           "-I", INCLUDE, "-I", CSRC, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
    return obj


def build(verbose: bool = False, extra_flags: list[str] | None = None, checked: bool = False) -> str:
    """Compile every source and link librolekv.so (or, checked=True,
    librolekv_checked.so with -DROLEKV_CHECKED); returns its path."""
    nvcc = nvcc_path()
    build_dir = CHECKED_BUILD_DIR if checked else BUILD_DIR
    lib_path = CHECKED_LIB_PATH if checked else LIB_PATH
    os.makedirs(build_dir, exist_ok=True)
    extra = list(extra_flags or []) + (["-DROLEKV_CHECKED"] if checked else [])
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(nvcc, s, extra, build_dir), SOURCES))
    tmp = lib_path + ".tmp"
    # (-ldl: the NVTX ranges find a profiler's injection library with dlopen)
    cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-ldl"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib_path)
    if verbose:
        print(f"built {lib_path}", file=sys.stderr)
    return lib_path


def build_all(verbose: bool = False) -> list[str]:
    """The plain and the checked library, built side by side."""
    with cf.ThreadPoolExecutor(max_workers=2) as ex:
        return list(ex.map(lambda c: build(verbose=verbose, checked=c), [False, True]))


if __name__ == "__main__":
    if sys.argv[1:] == ["--all"]:
        build_all(verbose=True)
    else:
        build(verbose=True, extra_flags=sys.argv[1:])
