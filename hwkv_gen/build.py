"""Build the seeded input generator: host fill (gcc) and device fill (nvcc, sm_103a)."""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
HOST_LIB = os.path.join(HERE, "libhwkv_gen_host.so")
DEV_LIB = os.path.join(HERE, "libhwkv_gen_dev.so")
HDR = os.path.join(HERE, "hwkv_gen.h")
HOST_SRC = os.path.join(HERE, "gen_host.c")
DEV_SRC = os.path.join(HERE, "gen_device.cu")


def host_command():
    return ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off", "-Wall",
            "-o", HOST_LIB, HOST_SRC]


def dev_command():
    return ["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo",
            "-std=c++17", "-Xcompiler", "-fPIC", "-shared", "-o", DEV_LIB, DEV_SRC]


def _stale(lib, deps):
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    return any(os.path.getmtime(p) > t for p in deps)


def jobs(force=False):
    """(command, output) pairs that need to run."""
    out = []
    if force or _stale(HOST_LIB, [HDR, HOST_SRC]):
        out.append((host_command(), HOST_LIB))
    if force or _stale(DEV_LIB, [HDR, DEV_SRC]):
        out.append((dev_command(), DEV_LIB))
    return out


def build(force=False, device=True):
    for cmd, lib in jobs(force):
        if lib == DEV_LIB and not device:
            continue
        subprocess.run(cmd, check=True)


if __name__ == "__main__":
    build(force="--force" in sys.argv)
