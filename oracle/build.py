"""Build the CPU oracle (plain C, fp64) into oracle/liboracle.so.

Test infrastructure: compiling the checker is part of the repository build;
only the tests, the smoke check and the benchmark's CPU-baseline leg load it.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
LIB = os.path.join(HERE, "liboracle.so")
SRC = [os.path.join(HERE, "hwkv_oracle.c")]
DEPS = SRC + [os.path.join(HERE, "..", "hwkv_gen", "hwkv_gen.h")]


def command():
    return ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
            "-Wall", "-Wno-unknown-pragmas", "-o", LIB] + SRC + ["-lm"]


def stale():
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(p) > t for p in DEPS)


def build(force=False):
    if force or stale():
        subprocess.run(command(), check=True)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv)
    print(LIB)
