"""Build the device-side payload filler (libro_workload.so) for sm_103a."""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "csrc", "payload_fill.cu")
LIB = os.path.join(HERE, "libro_workload.so")
HOST_SRC = os.path.join(HERE, "csrc", "payload_host.c")
HOST_LIB = os.path.join(HERE, "libro_workload_host.so")


def build_host(force: bool = False) -> str:
    """Host filler (plain C, gcc); needs no GPU toolchain."""
    if not force and os.path.exists(HOST_LIB) and os.path.getmtime(HOST_LIB) >= os.path.getmtime(HOST_SRC):
        return HOST_LIB
    tmp = HOST_LIB + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, HOST_SRC], check=True)
    os.replace(tmp, HOST_LIB)
    return HOST_LIB


def build(force: bool = False) -> str:
    build_host(force)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [nvcc, "-O3", "-std=c++17", "-shared", "-Xcompiler", "-fPIC", "-gencode",
           "arch=compute_103a,code=sm_103a", "-cudart", "static", "-o", tmp, SRC]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
