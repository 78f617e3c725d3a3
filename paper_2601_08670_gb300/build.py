"""In-tree build of libpced.so (the sm_103a decoding library) with nvcc.

Translation units compile in parallel, then link into one shared library
under ``paper_2601_08670_gb300/_lib``.  The library links the CUDA runtime
statically and fetches the driver's tensor-map encoder at run time, so it has
no link-time dependency on libcuda.
"""
from __future__ import annotations

import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
LIBDIR = os.path.join(HERE, "_lib")
LIB = os.path.join(LIBDIR, "libpced.so")
# the bounds-checked build: every guarded index outside its buffer sets
# PCED_DEV_BOUNDS in the status word and skips the access
CHECKED_LIBDIR = os.path.join(HERE, "_lib_checked")
CHECKED_LIB = os.path.join(CHECKED_LIBDIR, "libpced.so")
ROOT = os.path.dirname(HERE)
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
         "-I", os.path.join(ROOT, "include")]
SOURCES = ["attention.cu", "attention_noalloc.cu", "lm_head.cu", "select.cu", "adacad.cu", "aggregate.cu", "relevance.cu",
           "step.cu", "partition.cu", "host.cu"]


def _deps():
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(ROOT, "include", "pced.h")]
    return max(os.path.getmtime(f) for f in files)


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False, checked: bool = False) -> str:
    """Compiles libpced.so if a source is newer; `checked` builds the
    bounds-checked library (-DPCED_BOUNDS_CHECK) into its own folder."""
    libdir, lib = (CHECKED_LIBDIR, CHECKED_LIB) if checked else (LIBDIR, LIB)
    os.makedirs(libdir, exist_ok=True)
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= _deps():
        return lib
    procs = []
    objs = []
    for src in SOURCES:
        obj = os.path.join(libdir, src.replace(".cu", ".o"))
        objs.append(obj)
        cmd = ["nvcc", *ARCH, *FLAGS, *(["-DPCED_BOUNDS_CHECK"] if checked else []), "-c", os.path.join(CSRC, src),
               "-o", obj]
        if ptxas_info:
            cmd += ["-Xptxas", "-v"]
        procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
    failed = []
    for src, p in procs:
        out, _ = p.communicate()
        if verbose or p.returncode != 0:
            sys.stderr.write(f"--- {src}\n{out}")
        if p.returncode != 0:
            failed.append(src)
    if failed:
        raise RuntimeError(f"nvcc failed for {failed}")
    tmp = lib + f".tmp{os.getpid()}"
    subprocess.check_call(["nvcc", *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"])
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    build(force=True, verbose=True, ptxas_info="-v" in sys.argv)
