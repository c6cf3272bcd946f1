"""Builds libcurvadion.so in-tree: every csrc/*.cu compiled for sm_103a in parallel, then linked.

    python -m paper_2512_13728_gb300.build [--force]

The library is a plain C-ABI shared object (include/curvadion.h) linked against the shared
CUDA runtime; the driver API entry points it needs are fetched at run time, so loading it
needs no GPU.
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libcurvadion.so")
# the same sources with DION_DEBUG_CHECKS: workspace guards checked every step, tiles checked
BUILD_DEBUG = os.path.join(PKG, "_build_debug")
LIB_DEBUG = os.path.join(PKG, "libcurvadion_debug.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found")
    return cand


def cuda_lib_dir() -> str:
    home = os.environ.get("CUDA_HOME", os.path.dirname(os.path.dirname(os.path.realpath(nvcc()))))
    for d in ("lib64", "lib", "targets/sbsa-linux/lib", "targets/x86_64-linux/lib"):
        p = os.path.join(home, d)
        if os.path.exists(os.path.join(p, "libcudart.so")) or glob.glob(os.path.join(p, "libcudart.so*")):
            return p
    return os.path.join(home, "lib64")


def sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return (sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(CSRC, "*.h"))
            + [os.path.join(ROOT, "include", "curvadion.h"), os.path.abspath(__file__)])


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(d) <= t for d in _deps())


def build(force: bool = False, verbose: bool = False, debug: bool = False) -> str:
    """Builds libcurvadion.so, or with debug=True libcurvadion_debug.so (DION_DEBUG_CHECKS)."""
    LIB_OUT, BUILD_DIR = (LIB_DEBUG, BUILD_DEBUG) if debug else (LIB, BUILD)
    if not force and up_to_date(LIB_OUT):
        return LIB_OUT
    os.makedirs(BUILD_DIR, exist_ok=True)
    cc = nvcc()
    flags = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
                    "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include"), "-I", CSRC]
    if debug:
        flags += ["-DDION_DEBUG_CHECKS"]
    if os.environ.get("CURVADION_PTXAS_VERBOSE"):
        flags += ["-Xptxas", "-v"]
    procs, objs = [], []
    for src in sources():
        obj = os.path.join(BUILD_DIR, os.path.basename(src)[:-3] + ".o")
        objs.append(obj)
        cmd = [cc, "-c", src, "-o", obj] + flags
        procs.append((cmd, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
    failed = []
    for cmd, pr in procs:
        out, _ = pr.communicate()
        if verbose or pr.returncode != 0 or os.environ.get("CURVADION_PTXAS_VERBOSE"):
            sys.stderr.write(out)
        if pr.returncode != 0:
            failed.append(" ".join(cmd))
    if failed:
        raise RuntimeError("nvcc failed:\n" + "\n".join(failed))
    libdir = cuda_lib_dir()
    tmp = LIB_OUT + ".tmp"
    link = [cc, "-shared", "-o", tmp] + objs + ARCH + ["-cudart", "shared", "-L", libdir,
                                                        "-Xlinker", "-rpath," + libdir]
    r = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n" + r.stdout)
    os.replace(tmp, LIB_OUT)
    return LIB_OUT


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True, debug="--debug" in sys.argv))
