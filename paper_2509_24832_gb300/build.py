"""Builds the CUDA library libsemshare.so in-tree (paper_2509_24832_gb300/_lib/) with nvcc.

Every translation unit is compiled for sm_103a only, in parallel, then linked into one shared
library with the static CUDA runtime.  No cmake, no torch extension machinery."""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIBDIR = os.path.join(PKG, "_lib")
LIB = os.path.join(LIBDIR, "libsemshare.so")
SOURCES = ["api.cu", "hash.cu", "hash_2sm.cu", "match.cu", "match_tc.cu", "gather.cu", "deviation.cu", "fetch.cu"]
# measurement support, linked into a library of its own so that libsemshare.so exports only the
# entry points of include/semshare.h
PROBE_SOURCES = ["probe.cu"]
PROBE_LIB = os.path.join(LIBDIR, "libsemshare_probe.so")
# the same sources with -DSEMSHARE_CHECKED: kernels that also verify their pipeline bookkeeping
CHECKED_LIB = os.path.join(LIBDIR, "libsemshare_checked.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
# -warn-spills: a register spill in a file with tensor-memory loads is a build error (below).  Those
# kernels hand tcgen05.ld destination registers to later code before the load's wait; a spill placed
# in between would store them before the data arrives.
NO_SPILL = {"hash.cu", "hash_2sm.cu", "match_tc.cu"}
NVCC_FLAGS = ARCH + ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-O2", "-Xptxas", "-warn-spills",
                     "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libsemshare.so")
    return path


def _inputs():
    return [os.path.join(CSRC, s) for s in SOURCES + PROBE_SOURCES] + glob.glob(os.path.join(CSRC, "*.cuh")) + \
        glob.glob(os.path.join(INCLUDE, "*.h")) + [os.path.abspath(__file__)]


def up_to_date() -> bool:
    if not all(os.path.exists(p) for p in (LIB, PROBE_LIB, CHECKED_LIB)):
        return False
    t = min(os.path.getmtime(p) for p in (LIB, PROBE_LIB, CHECKED_LIB))
    return all(os.path.getmtime(p) <= t for p in _inputs())


def build(force: bool = False, verbose: bool = False, extra_flags: list[str] | None = None) -> str:
    """Compile and link libsemshare.so, the measurement probe library libsemshare_probe.so and the
    checked build libsemshare_checked.so; returns the path of libsemshare.so.  No-op when up to
    date."""
    if not force and not extra_flags and up_to_date():
        return LIB
    os.makedirs(os.path.join(LIBDIR, "obj"), exist_ok=True)
    os.makedirs(os.path.join(LIBDIR, "obj_checked"), exist_ok=True)
    cc = nvcc()
    flags = NVCC_FLAGS + list(extra_flags or [])
    procs = []
    objs = []
    jobs = [(src, "obj", []) for src in SOURCES + PROBE_SOURCES] + \
        [(src, "obj_checked", ["-DSEMSHARE_CHECKED"]) for src in SOURCES]
    for src, sub, defs in jobs:
        obj = os.path.join(LIBDIR, sub, src.replace(".cu", ".o"))
        objs.append(obj)
        cmd = [cc, *flags, *defs, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            print(" ".join(cmd), file=sys.stderr)
        procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
    failed = []
    for src, p in procs:
        out, _ = p.communicate()
        spilled = src in NO_SPILL and "spill" in (out or "").lower()
        if out and (verbose or p.returncode or spilled):
            print(out, file=sys.stderr)
        if p.returncode or spilled:
            failed.append(src)
    if failed:
        raise RuntimeError(f"nvcc failed (or spilled registers) on {failed}")
    n, m = len(SOURCES), len(SOURCES) + len(PROBE_SOURCES)
    for lib, parts in ((LIB, objs[:n]), (PROBE_LIB, objs[n:m]), (CHECKED_LIB, objs[m:])):
        tmp = lib + f".tmp{os.getpid()}"
        subprocess.run([cc, *ARCH, "-shared", "-Xcompiler", "-fPIC", *parts, "-o", tmp], check=True)
        os.replace(tmp, lib)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
