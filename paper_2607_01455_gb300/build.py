"""Compile libember.so (the CUDA library behind include/ember.h) for sm_103a.

Each .cu file compiles to an object in parallel, then nvcc links the shared
library in place under paper_2607_01455_gb300/_lib/.  nvcc cross-compiles, so
this runs on a machine without a GPU too.
"""
import concurrent.futures
import os
import subprocess
import tempfile

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB_DIR = os.path.join(PKG, "_lib")
LIB = os.path.join(LIB_DIR, "libember.so")

NVCC = os.environ.get("NVCC", "nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2",
         "-I", INCLUDE, "-I", CSRC, "--expt-relaxed-constexpr"]


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _deps():
    return sources() + [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".h")] + \
        [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h")]


def _compile(src, extra, objdir):
    obj = os.path.join(objdir, os.path.basename(src)[:-3] + ".o")
    subprocess.run([NVCC, *ARCH, *FLAGS, *extra, "-c", src, "-o", obj], check=True)
    return obj


def build_library(force: bool = False, verbose_ptxas: bool = False) -> str:
    """Build libember.so unless it is newer than every source and header."""
    if (not force and not verbose_ptxas and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= max(os.path.getmtime(p) for p in _deps())):
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    os.makedirs(LIB_DIR, exist_ok=True)
    extra = ["-Xptxas", "-v"] if verbose_ptxas else []
    # objects of concurrent builds (parallel test workers) never collide
    with tempfile.TemporaryDirectory(dir=BUILD) as objdir:
        with concurrent.futures.ThreadPoolExecutor(max_workers=len(sources())) as ex:
            objs = list(ex.map(lambda s: _compile(s, extra, objdir), sources()))
        tmp = LIB + f".tmp{os.getpid()}"
        subprocess.run([NVCC, *ARCH, "-shared", "-o", tmp, *objs], check=True)
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    import sys
    print(build_library(force=True, verbose_ptxas="-v" in sys.argv))
