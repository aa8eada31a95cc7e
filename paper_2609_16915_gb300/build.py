"""Build librosetta.so in-tree for sm_103a (nvcc only, no cmake).

Each translation unit is compiled in parallel, then linked into
``paper_2609_16915_gb300/librosetta.so``.
"""

from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
ROOT = os.path.dirname(HERE)
LIB = os.path.join(HERE, "librosetta.so")
DEBUG_LIB = os.path.join(HERE, "librosetta_debug.so")
BUILD_DIR = os.path.join(ROOT, "_build")
SOURCES = ["tables.cu", "bsk_transform.cu", "blind_rotate.cu", "blind_rotate3.cu", "keyswitch.cu", "keyswitch_tc.cu",
           "rosetta_api.cu", "pbs_noalloc.cu", "trace.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build librosetta")


def _flags(verbose: bool):
    f = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include")] + ARCH
    if verbose:
        f += ["-Xptxas", "-v"]
    return f


def _stale(objs, lib) -> bool:
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f != PEAKS_SRC] + [os.path.join(ROOT, "include", "rosetta.h"),
                                                                                 __file__]
    return any(os.path.getmtime(d) > t for d in deps)


PEAKS_SRC = "int_peaks.cu"
PEAKS_LIB = os.path.join(HERE, "libintpeaks.so")


def build_peaks(force: bool = False) -> str:
    """libintpeaks.so: the integer issue-rate microbenchmarks bench.py runs
    (a separate library, not part of the PBS path)."""
    src = os.path.join(CSRC, PEAKS_SRC)
    if not force and os.path.exists(PEAKS_LIB) and os.path.getmtime(PEAKS_LIB) >= max(os.path.getmtime(src),
                                                                                     os.path.getmtime(__file__)):
        return PEAKS_LIB
    tmp = PEAKS_LIB + f".tmp{os.getpid()}"
    cmd = [nvcc(), "-shared", "-o", tmp, src] + _flags(False) + ["-lcudart"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {PEAKS_SRC}:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, PEAKS_LIB)
    return PEAKS_LIB


def build(force: bool = False, verbose: bool = False, debug: bool = False) -> str:
    """Build librosetta.so, or with debug=True librosetta_debug.so: the same
    sources compiled with -DROSETTA_DEBUG (device-side bounds checks that
    report ROSETTA_ERR_BOUNDS instead of reading outside a buffer)."""
    lib = DEBUG_LIB if debug else LIB
    bdir = os.path.join(BUILD_DIR, "debug") if debug else BUILD_DIR
    os.makedirs(bdir, exist_ok=True)
    objs = [os.path.join(bdir, s.replace(".cu", ".o")) for s in SOURCES]
    if not force and not _stale(objs, lib):
        return lib
    cc = nvcc()
    extra = ["-DROSETTA_DEBUG"] if debug else []

    def compile_one(src_obj):
        src, obj = src_obj
        cmd = [cc, "-c", os.path.join(CSRC, src), "-o", obj] + _flags(verbose) + extra
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return r.stderr

    with ThreadPoolExecutor(len(SOURCES)) as ex:
        logs = list(ex.map(compile_one, zip(SOURCES, objs)))
    if verbose:
        for s, log in zip(SOURCES, logs):
            print(f"--- {s}\n{log}")
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [cc, "-shared", "-o", tmp] + objs + ARCH + ["-lcudart"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    import sys
    print(build(force=True, verbose="-v" in sys.argv, debug="--debug" in sys.argv))
