"""Build the CUDA library libbandlu.so in-tree (sm_103a only).

Each .cu under csrc/ is compiled to an object in parallel with nvcc, then the
objects are linked into ``_build/libbandlu.so`` next to this file.  The CUDA
runtime is linked statically, so the library depends only on the driver.
"""
from __future__ import annotations

import concurrent.futures as cf
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
LIB = os.path.join(BUILD, "libbandlu.so")
# Checked variant for development and tests: inter-warp hand-offs use bounded
# mbarrier waits (a protocol slip ends a kernel with an error status instead of
# a hang).  Never the library the product path loads.
CHECKED_LIB = os.path.join(BUILD, "libbandlu_checked.so")
# Traced variant for development and profiling: the wide-band chain kernel records the global
# timer at its panel boundaries and waits (include/bandlu_trace.h).  Never the library the
# product path loads.
TRACE_LIB = os.path.join(BUILD, "libbandlu_trace.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC,
              "--expt-relaxed-constexpr"]


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found: the CUDA library cannot be built")
    return path


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _deps() + [os.path.abspath(__file__)])


def build(force: bool = False, verbose: bool = False, extra_flags: list[str] | None = None,
          checked: bool = False, trace: bool = False) -> str:
    """Compile and link the library (or its checked or traced variant); returns its path.
    Raises on a compiler error."""
    lib = CHECKED_LIB if checked else (TRACE_LIB if trace else LIB)
    if not force and up_to_date(lib):
        return lib
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    flags = NVCC_FLAGS + list(extra_flags or []) + (["-DBANDLU_BOUNDED_SYNC"] if checked else []) + \
        (["-DBANDLU_TRACE"] if trace else [])
    suffix = ".checked.o" if checked else (".trace.o" if trace else ".o")

    def compile_one(src: str) -> str:
        obj = os.path.join(BUILD, os.path.basename(src)[:-3] + suffix)
        cmd = [cc, *ARCH, *flags, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout + r.stderr, file=sys.stderr)
        return obj

    srcs = _sources()
    with cf.ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        objs = list(ex.map(compile_one, srcs))
    tmp = lib + f".tmp{os.getpid()}"
    r = subprocess.run([cc, *ARCH, "-shared", "-o", tmp, *objs], capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                extra_flags=["-Xptxas", "-v"] if "--ptxas-v" in sys.argv else None,
                checked="--checked" in sys.argv, trace="--trace" in sys.argv))
