"""Builds libcm.so in-tree (next to this file) for sm_103a with nvcc and g++.

Three translation units compiled in parallel, then one shared-library link:
  csrc/cm_host.cpp       host core (g++, C++17, no floating-point contraction)
  csrc/blake2s_tree.cu   content-address kernels (nvcc, sm_103a)
  csrc/render.cu         render kernel (nvcc, sm_103a)
  csrc/dedup.cu          byte comparison of the re-delivery fast path (nvcc, sm_103a)
  csrc/readback.cu       small device-to-host results written by the SMs (nvcc, sm_103a)
The CUDA runtime is linked statically into libcm.so and only the cm_* symbols
are exported (csrc/libcm.map).

`--bounds` (build(bounds=True)) builds the same sources with -DCM_DEBUG_BOUNDS into
libcm_bounds.so (objects in _build_bounds/): a testing build whose kernels check every
global access against its buffer (csrc/cm_bounds.h). The binding loads it when the
environment variable CM_LIBRARY names it.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
REPO_DIR = os.path.dirname(PKG_DIR)
CSRC = os.path.join(PKG_DIR, "csrc")
INCLUDE = os.path.join(REPO_DIR, "include")
BUILD_DIR = os.path.join(PKG_DIR, "_build")
LIB_PATH = os.path.join(PKG_DIR, "libcm.so")
BOUNDS_BUILD_DIR = os.path.join(PKG_DIR, "_build_bounds")
BOUNDS_LIB_PATH = os.path.join(PKG_DIR, "libcm_bounds.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-std=c++17", "-O3", "-lineinfo", "-fmad=false", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-ffp-contract=off", "-I" + INCLUDE, "-I" + CSRC]
CXX_FLAGS = ["-std=c++17", "-O2", "-fPIC", "-ffp-contract=off", "-Wall", "-Wextra",
             "-I" + INCLUDE, "-I" + CSRC]

CUDA_SOURCES = ["blake2s_tree.cu", "render.cu", "dedup.cu", "readback.cu"]
CXX_SOURCES = ["cm_host.cpp"]


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home:
        return home
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return "/usr/local/cuda"


def _run(cmd, verbose):
    if verbose:
        print(" ".join(cmd), flush=True)
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError("build step failed:\n" + " ".join(cmd) + "\n" + r.stdout)
    return r.stdout


def build(verbose: bool = False, ptxas_info: bool = False, bounds: bool = False) -> str:
    """Compile and link libcm.so (libcm_bounds.so with bounds=True); returns its path.
    Raises RuntimeError on failure."""
    build_dir = BOUNDS_BUILD_DIR if bounds else BUILD_DIR
    lib_path = BOUNDS_LIB_PATH if bounds else LIB_PATH
    defs = ["-DCM_DEBUG_BOUNDS"] if bounds else []
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    if not os.path.exists(nvcc):
        nvcc = shutil.which("nvcc") or "nvcc"
    cxx = os.environ.get("CXX", shutil.which("g++") or "g++")
    os.makedirs(build_dir, exist_ok=True)
    cuda_inc = os.path.join(cuda, "include")
    jobs = []
    for src in CUDA_SOURCES:
        obj = os.path.join(build_dir, src + ".o")
        extra = ["-Xptxas", "-v"] if ptxas_info else []
        jobs.append([nvcc] + ARCH + NVCC_FLAGS + defs + extra + ["-c", os.path.join(CSRC, src), "-o", obj])
    for src in CXX_SOURCES:
        obj = os.path.join(build_dir, src + ".o")
        jobs.append([cxx] + CXX_FLAGS + defs + ["-I" + cuda_inc, "-c", os.path.join(CSRC, src), "-o", obj])
    with ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        logs = list(ex.map(lambda c: _run(c, verbose), jobs))
    if ptxas_info:
        for log in logs:
            print(log)
    objs = [os.path.join(build_dir, s + ".o") for s in CUDA_SOURCES + CXX_SOURCES]
    tmp = lib_path + ".tmp"
    link = ["-shared", "-Xcompiler", "-fPIC", "-cudart", "static",
            "-Xlinker", "--version-script=" + os.path.join(CSRC, "libcm.map"),
            "-Xlinker", "-Bsymbolic"]
    _run([nvcc] + ARCH + link + ["-o", tmp] + objs, verbose)
    os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    import sys
    print(build(verbose=True, ptxas_info="--ptxas" in sys.argv, bounds="--bounds" in sys.argv))
