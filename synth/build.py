"""Build the seeded input generator: libsynth_host.so (C) and, for GPU runs,
libsynth_dev.so (CUDA, sm_103a).  Both compile synth_core.h with floating-point
contraction off so that they produce bit-identical values.

    python -m synth.build
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CORE = os.path.join(HERE, "synth_core.h")
HOST_SRC = os.path.join(HERE, "synth_host.c")
DEV_SRC = os.path.join(HERE, "synth_dev.cu")
HOST_LIB = os.path.join(HERE, "libsynth_host.so")
DEV_LIB = os.path.join(HERE, "libsynth_dev.so")
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")


def _stale(lib, srcs):
    return not os.path.exists(lib) or os.path.getmtime(lib) < max(
        os.path.getmtime(s) for s in srcs + [__file__])


def _run(cmd, what):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"{what} failed:\n{r.stdout}\n{r.stderr}")


def build_host(force=False):
    if force or _stale(HOST_LIB, [HOST_SRC, CORE]):
        tmp = HOST_LIB + ".tmp"
        _run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-pthread",
              HOST_SRC, "-o", tmp, "-lm"], "gcc")
        os.replace(tmp, HOST_LIB)
    return HOST_LIB


def build_dev(force=False):
    if force or _stale(DEV_LIB, [DEV_SRC, CORE]):
        tmp = DEV_LIB + ".tmp"
        _run([NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "--fmad=false",
              "-Xcompiler", "-fPIC", "-shared", DEV_SRC, "-o", tmp], "nvcc")
        os.replace(tmp, DEV_LIB)
    return DEV_LIB


def build(force=False):
    return build_host(force), build_dev(force)


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
