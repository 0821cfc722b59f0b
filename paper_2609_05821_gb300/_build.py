"""Builds libconduit.so in-tree from csrc/*.cu for sm_103a (nvcc, no cmake).

Each translation unit compiles in parallel into _build/, then nvcc links the
shared library next to this file. A unit is rebuilt only when it or a header
is newer than its object.
"""

from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libconduit.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include"), "-I", CSRC]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libconduit.so")


def _headers_mtime() -> float:
    hs = glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(ROOT, "include", "*.h"))
    return max((os.path.getmtime(h) for h in hs), default=0.0)


def build(verbose: bool = False, extra_flags=(), variant: str = "") -> str:
    """Compile every csrc/*.cu and link libconduit.so; returns its path.

    A `variant` builds a separate library (libconduit_<variant>.so, objects in
    _build_<variant>/) with `extra_flags`, for the test suite only."""
    nvcc = _nvcc()
    bdir = os.path.join(HERE, "_build_" + variant) if variant else BUILD
    lib = os.path.join(HERE, f"libconduit_{variant}.so") if variant else LIB
    os.makedirs(bdir, exist_ok=True)
    sources = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    hdr_t = _headers_mtime()

    def compile_one(src: str) -> str:
        obj = os.path.join(bdir, os.path.basename(src)[:-3] + ".o")
        if os.path.exists(obj) and os.path.getmtime(obj) >= max(os.path.getmtime(src), hdr_t):
            return obj
        cmd = [nvcc, *ARCH, *FLAGS, *extra_flags, "-c", src, "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed on {os.path.basename(src)}:\n{res.stderr}")
        if verbose and res.stderr:
            print(res.stderr, flush=True)
        return obj

    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        objs = list(ex.map(compile_one, sources))
    if not os.path.exists(lib) or os.path.getmtime(lib) < max(os.path.getmtime(o) for o in objs):
        cmd = [nvcc, *ARCH, "-shared", "-o", lib, *objs]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"link of {os.path.basename(lib)} failed:\n{res.stderr}")
    return lib


def build_test_hooks(verbose: bool = False) -> str:
    """The test-only library libconduit_testhooks.so: bounded device waits give
    up after 1 ms instead of 1 s, and conduit_test_withhold_v_tile(n) makes the
    scoring kernel's V producer skip one tile (no copy, no arrive), so a test
    can run the timeout path without a fault. Never loaded by the package."""
    return build(verbose, ("-DCONDUIT_TEST_HOOKS", "-DCONDUIT_WAIT_NS=1000000ull"), "testhooks")


if __name__ == "__main__":
    print(build(verbose=True))
