"""Build the CPU oracle (TEST INFRASTRUCTURE ONLY): gcc -O2 -fopenmp, no CUDA.

The oracle library is compiled on whichever machine runs the tests (x86_64 here, aarch64
on the GPU host); `-ffp-contract=off` keeps its fp64 results identical on both.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "jf_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libjforacle.so")


def build(force: bool = False) -> str:
    """Compile oracle/jf_oracle.c into oracle/_build/libjforacle.so; returns the path."""
    os.makedirs(OUT_DIR, exist_ok=True)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-ffp-contract=off",
           "-Wall", "-Wno-unused-function", "-o", tmp, SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
