"""Build libhwkv.so (the C-ABI library of include/hwkv.h) for sm_103a, in-tree.

Each translation unit is compiled by nvcc in parallel, then linked with
`nvcc -shared`. No cmake; a rebuild happens only when a source or header is
newer than the library.
"""
import glob
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OBJ = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libhwkv.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
         "--expt-relaxed-constexpr", "-I" + os.path.join(ROOT, "include")]


def sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def deps():
    return sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + [
        os.path.join(ROOT, "include", "hwkv.h")]


def stale():
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(p) > t for p in deps())


def compile_jobs(extra=()):
    os.makedirs(OBJ, exist_ok=True)
    jobs = []
    for src in sources():
        obj = os.path.join(OBJ, os.path.basename(src)[:-3] + ".o")
        jobs.append((["nvcc"] + ARCH + FLAGS + list(extra) + ["-c", src, "-o", obj], obj))
    return jobs


def link_command(objs):
    return ["nvcc"] + ARCH + ["-shared", "-o", LIB] + objs + ["-lcuda"]


def build(force=False, verbose=False):
    if not (force or stale()):
        return LIB
    jobs = compile_jobs(["-Xptxas", "-v"] if verbose else [])
    procs = [(subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT), cmd)
             for cmd, _ in jobs]
    failed = []
    for p, cmd in procs:
        out, _ = p.communicate()
        if verbose or p.returncode != 0:
            sys.stdout.write(out.decode(errors="replace"))
        if p.returncode != 0:
            failed.append(cmd[-3])
    if failed:
        raise RuntimeError("nvcc failed for: " + ", ".join(failed))
    subprocess.run(link_command([o for _, o in jobs]), check=True)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose="-v" in sys.argv)
    print(LIB)
