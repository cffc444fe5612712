"""Build ``libdqgan.so`` (the sm_103a CUDA library behind include/dqgan.h).

Each ``csrc/*.cu`` translation unit is compiled by nvcc in parallel for
``sm_103a`` only, with ``-fmad=false`` (no fused multiply-add anywhere: the
method's arithmetic must round once per operation) and ``-lineinfo``, then
linked into a shared library next to this file.  The CUDA runtime is linked
statically so the library does not depend on the runtime a host program
loads.
"""
from __future__ import annotations

import concurrent.futures
import glob
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIBRARY = os.path.join(HERE, "libdqgan.so")
# The checked build: the same sources with -DDQGAN_CHECK_BOUNDS (index checks
# that skip an out-of-range access and report it, guard zones around the
# top-k scratch), for the tests; the binding loads it when DQGAN_LIBRARY
# names it.
CHECKED_LIBRARY = os.path.join(HERE, "libdqgan_checked.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-fmad=false", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-fvisibility=hidden", "--expt-relaxed-constexpr"]


def nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: the DQGAN CUDA library cannot be built")
    return cand


def sources() -> list[str]:
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _inputs() -> list[str]:
    return sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + [os.path.join(INCLUDE, "dqgan.h"),
                                                                  os.path.abspath(__file__)]


def up_to_date(library: str = LIBRARY) -> bool:
    if not os.path.exists(library):
        return False
    t = os.path.getmtime(library)
    return all(os.path.getmtime(p) <= t for p in _inputs())


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False, checked: bool = False) -> str:
    """Compile and link the library (or, with checked=True, the checked
    build) if any input changed; return its path."""
    library = CHECKED_LIBRARY if checked else LIBRARY
    build_dir = BUILD_DIR + ("_checked" if checked else "")
    if not force and up_to_date(library):
        return library
    os.makedirs(build_dir, exist_ok=True)
    exe = nvcc()
    extra = ["-Xptxas", "-v"] if ptxas_info else []
    if checked:
        extra.append("-DDQGAN_CHECK_BOUNDS")

    def compile_one(src: str) -> tuple[str, str]:
        obj = os.path.join(build_dir, os.path.basename(src).replace(".cu", ".o"))
        cmd = [exe, *ARCH, *NVCC_FLAGS, *extra, "-I", INCLUDE, "-I", CSRC, "-c", src, "-o", obj]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed on {os.path.basename(src)}:\n{res.stderr}")
        return obj, res.stderr

    with concurrent.futures.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 4)) as ex:
        results = list(ex.map(compile_one, sources()))
    if verbose or ptxas_info:
        for _, log in results:
            if log.strip():
                print(log)
    tmp = library + f".tmp{os.getpid()}"
    cmd = [exe, *ARCH, "-shared", "-o", tmp, *[o for o, _ in results], "-cudart", "static"]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"nvcc link failed:\n{res.stderr}")
    os.replace(tmp, library)
    return library


if __name__ == "__main__":
    import sys
    print(build(force=True, verbose=True, ptxas_info="-v" in sys.argv))
