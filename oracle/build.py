"""Compile the CPU oracle (ember_oracle.c) into a shared library with gcc.

Test infrastructure only: the oracle checks the CUDA library, it is never part
of it.  The flags keep every floating-point operation as written: no fast-math,
no contraction of a*b+c into a fused multiply-add.
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "ember_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libember_oracle.so")

CFLAGS = ["-O2", "-std=c11", "-fno-fast-math", "-ffp-contract=off",
          "-fPIC", "-shared", "-Wall", "-Wextra", "-Wno-unknown-pragmas"]


LIB_OMP = os.path.join(OUT_DIR, "libember_oracle_omp.so")


def build_oracle(force: bool = False, openmp: bool = False) -> str:
    """Build the oracle library if it is missing or older than its source.
    openmp=True builds the all-cores copy the CPU baseline times (same
    source, -fopenmp; the same results bit for bit)."""
    os.makedirs(OUT_DIR, exist_ok=True)
    lib = LIB_OMP if openmp else LIB
    if (not force and os.path.exists(lib)
            and os.path.getmtime(lib) >= os.path.getmtime(SRC)):
        return lib
    tmp = lib + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *CFLAGS, *(["-fopenmp"] if openmp else []), "-o", tmp, SRC, "-lm"], check=True)
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build_oracle(force=True))
    print(build_oracle(force=True, openmp=True))
