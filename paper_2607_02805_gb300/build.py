"""Build libbdscan.so in-tree with nvcc for sm_103a (GB300).

Each .cu file is compiled to an object in parallel, then linked into
``paper_2607_02805_gb300/lib/libbdscan.so``. The CUDA runtime is linked
statically, so the library needs only the driver at run time. A rebuild
happens when any source or header is newer than the library.

The debug build, ``lib/libbdscan_debug.so``, is the same sources compiled
with ``-DBDSCAN_DEBUG=1``: its kernels check their extents and write device
status words, and its entry points return BDSCAN_ERR_DEVICE when a check
failed (include/bdscan.h). ``build_all()`` compiles both variants at once.
"""

from __future__ import annotations

import concurrent.futures
import glob
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIBDIR = os.path.join(HERE, "lib")
LIB = os.path.join(LIBDIR, "libbdscan.so")
LIB_DEBUG = os.path.join(LIBDIR, "libbdscan_debug.so")
DEBUG_FLAGS = ["-DBDSCAN_DEBUG=1"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-I" + INCLUDE, "-I" + CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA library cannot be built")


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + sorted(glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(CSRC, "*.h"))
                               + glob.glob(os.path.join(INCLUDE, "*.h")) + [os.path.abspath(__file__)])


def up_to_date(debug: bool = False) -> bool:
    lib = LIB_DEBUG if debug else LIB
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _deps())


def _variants(debug_list, force):
    return [d for d in debug_list if force or not up_to_date(d)]


def _build_variants(debug_list, verbose=False, extra_flags=()):
    """Compiles every (variant, source) pair in one process pool, then links."""
    os.makedirs(LIBDIR, exist_ok=True)
    cc = nvcc()
    srcs = _sources()
    jobs = []
    for dbg in debug_list:
        bdir = os.path.join(BUILD, "debug") if dbg else BUILD
        os.makedirs(bdir, exist_ok=True)
        flags = list(extra_flags) + (DEBUG_FLAGS if dbg else [])
        for src in srcs:
            jobs.append((dbg, src, os.path.join(bdir, os.path.basename(src)[:-3] + ".o"), flags))

    def compile_one(job):
        _, src, obj, flags = job
        cmd = [cc] + ARCH + NVCC_FLAGS + flags + ["-c", src, "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {os.path.basename(src)} {' '.join(flags)}:\n{r.stdout}\n{r.stderr}")
        return r.stdout + r.stderr

    with concurrent.futures.ThreadPoolExecutor(max_workers=max(1, len(jobs))) as ex:
        logs = list(ex.map(compile_one, jobs))
    if verbose:
        for job, log in zip(jobs, logs):
            sys.stdout.write(f"== {os.path.basename(job[1])} {' '.join(job[3])}\n{log}")
    out = []
    for dbg in debug_list:
        lib = LIB_DEBUG if dbg else LIB
        objs = [j[2] for j in jobs if j[0] == dbg]
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [cc] + ARCH + ["-shared", "-o", tmp] + objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
        out.append(lib)
    return out


def build(force: bool = False, verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    """Builds one variant (the release library, or the debug one) if stale."""
    if _variants([debug], force):
        _build_variants([debug], verbose, extra_flags)
    return LIB_DEBUG if debug else LIB


def build_all(force: bool = False, verbose: bool = False) -> list:
    """Builds the release and the debug library (whichever is stale) in one pool."""
    todo = _variants([False, True], force)
    if todo:
        _build_variants(todo, verbose)
    return [LIB, LIB_DEBUG]


if __name__ == "__main__":
    for p in build_all(force="--force" in sys.argv, verbose="-v" in sys.argv):
        print(p)
