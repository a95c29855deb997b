"""Build ``libfrt.so`` in-tree with nvcc for sm_103a (no torch extension machinery).

Each ``csrc/*.cu`` is compiled to an object in parallel, then linked into a shared
library exporting the C ABI of ``include/frt.h`` and ``include/frt_selftest.h``.
"""

from __future__ import annotations

import concurrent.futures as cf
import os
import platform
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libfrt.so")
# the FRT_DEBUG variant: kernels bounds-check every derived index and record
# FRT_ERR_BOUNDS instead of touching memory outside its buffer; every stream sync also
# compares the guard words around the KV cache
DEBUG_BUILD = os.path.join(PKG, "_build_debug")
DEBUG_LIB = os.path.join(PKG, "libfrt_debug.so")
ARCH_FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a"]
CFLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
          "-I", os.path.join(ROOT, "include"), "--expt-relaxed-constexpr"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libfrt.so")


def sources() -> list[str]:
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _inputs() -> list[str]:
    files = sources()
    files += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    inc = os.path.join(ROOT, "include")
    files += [os.path.join(inc, f) for f in os.listdir(inc) if f.endswith(".h")]
    return files


def _stamp(debug: bool = False) -> str:
    return f"{platform.machine()}|{' '.join(ARCH_FLAGS + CFLAGS)}|{'debug' if debug else ''}"


def up_to_date(debug: bool = False) -> bool:
    build_dir, lib = (DEBUG_BUILD, DEBUG_LIB) if debug else (BUILD, LIB)
    stamp = os.path.join(build_dir, "stamp")
    if not (os.path.exists(lib) and os.path.exists(stamp)):
        return False
    if open(stamp).read() != _stamp(debug):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    """Compile and link libfrt.so (libfrt_debug.so with debug=True, compiled with
    -DFRT_DEBUG); returns its path. Raises on a compiler error."""
    BUILD, LIB = (DEBUG_BUILD, DEBUG_LIB) if debug else (globals()["BUILD"], globals()["LIB"])
    if debug:
        extra_flags = ("-DFRT_DEBUG", *extra_flags)
    if not force and (debug or not extra_flags) and up_to_date(debug):
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()

    def compile_one(src: str) -> str:
        obj = os.path.join(BUILD, os.path.basename(src)[:-3] + ".o")
        cmd = [cc, *ARCH_FLAGS, *CFLAGS, *extra_flags, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {os.path.basename(src)}:\n{r.stderr}")
        if verbose and r.stderr:
            print(r.stderr)
        return obj

    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 2)) as ex:
        objs = list(ex.map(compile_one, sources()))
    tmp = LIB + ".tmp"
    r = subprocess.run([cc, *ARCH_FLAGS, "-shared", "-o", tmp, *objs], capture_output=True,
                       text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(os.path.join(BUILD, "stamp"), "w") as f:
        f.write(_stamp(debug))
    return LIB


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose=True,
                extra_flags=("-Xptxas", "-v") if "--ptxas" in sys.argv else (),
                debug="--debug" in sys.argv))
