"""Builds the fp64 oracle's shared library with gcc (test infrastructure).

Usage: ``python -m oracle.build`` or ``oracle.build.build()``. The output,
``oracle/_smem_oracle.so``, is a build artefact (git-ignored) and is rebuilt
on each machine, since the GPU host is a different architecture.
"""
from __future__ import annotations

import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "smem_oracle.c")
LIB = os.path.join(HERE, "_smem_oracle.so")


def build(force: bool = False) -> str:
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c99", "-O2", "-fPIC", "-shared", "-fno-fast-math", SRC, "-o", tmp, "-lm"]
    # OpenMP spreads heads over threads (the arithmetic of a head is the
    # same either way); without libgomp the library builds single-threaded
    r = subprocess.run(cmd[:-3] + ["-fopenmp"] + cmd[-3:], capture_output=True)
    if r.returncode != 0:
        subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
