"""Build ``libloca.so`` in-tree with nvcc for sm_103a (GB300).

Each CUDA translation unit is compiled in parallel to ``_build/*.o`` and linked into
``paper_2608_03020_gb300/libloca.so``.  The build is skipped when the library is newer than
every source and header.  ``build(debug=True)`` makes ``libloca_debug.so`` (objects in
``_build_debug/``) with ``-DLOCA_DEBUG``: the same entry points with index bounds checks in
every kernel (``csrc/debug_check.cuh``).
"""

from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libloca.so")
LIB_DEBUG = os.path.join(PKG, "libloca_debug.so")
BUILD_DEBUG = os.path.join(PKG, "_build_debug")
SOURCES = ["loca_abi.cu", "error.cu", "targets.cu", "stats.cu", "gram_tc.cu", "solve.cu", "calib.cu",
           "noalloc.cu", "host_mem.cu", "kspace.cu", "align.cu", "calib_rsvd.cu",
           "targets_sq.cu", "project_tc.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVFLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
                  "-I" + os.path.join(ROOT, "include")]


def _nvcc() -> str:
    exe = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(exe):
        raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build libloca.so")
    return exe


def _inputs():
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cu", ".h", ".cuh"))]
    files.append(os.path.join(ROOT, "include", "loca.h"))
    files.append(os.path.abspath(__file__))
    return files


def up_to_date(debug: bool = False) -> bool:
    lib = LIB_DEBUG if debug else LIB
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False, debug: bool = False) -> str:
    """Compile and link the library (the LOCA_DEBUG variant when ``debug``); returns its path."""
    lib, bdir = (LIB_DEBUG, BUILD_DEBUG) if debug else (LIB, BUILD)
    if not force and up_to_date(debug):
        return lib
    nvcc = _nvcc()
    os.makedirs(bdir, exist_ok=True)
    extra = ["-Xptxas", "-v"] if ptxas_info else []
    if debug:
        extra.append("-DLOCA_DEBUG")

    def compile_one(src):
        obj = os.path.join(bdir, src.replace(".cu", ".o"))
        cmd = [nvcc, *NVFLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with cf.ThreadPoolExecutor(max_workers=min(len(SOURCES), os.cpu_count() or 4)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose or ptxas_info:
        for _, log in results:
            if log.strip():
                print(log)
    tmp = lib + ".tmp"
    cmd = [nvcc, *ARCH, "-shared", "--cudart", "shared", "-o", tmp] + [o for o, _ in results]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    import sys

    print(build(force="--force" in sys.argv, verbose=True, ptxas_info="--ptxas" in sys.argv,
                debug="--debug" in sys.argv))
