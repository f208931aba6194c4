"""Builds libsmem.so (the C ABI of include/smem.h) for sm_103a with nvcc.

Each translation unit compiles in its own nvcc process, in parallel; the
objects link into ``paper_2609_32395_gb300/libsmem.so`` (git-ignored). The
library links the shared CUDA runtime, so inside a process that already
loaded PyTorch it shares PyTorch's runtime and streams.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OBJ = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libsmem.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
SOURCES = ["smem_capi.cpp", "smem_copy.cu", "smem_decode.cu", "smem_gemm.cu", "smem_prefill.cu", "smem_recompute.cu"]
HEADERS = ["smem_device.cuh", "smem_internal.h", "smem_tc.cuh"]


def _nvcc() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home and os.path.exists(os.path.join(home, "bin", "nvcc")):
        return os.path.join(home, "bin", "nvcc")
    found = shutil.which("nvcc")
    if found:
        return found
    return "/usr/local/cuda/bin/nvcc"


def _cuda_lib_dir(nvcc: str) -> str:
    return os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(nvcc))), "lib64")


def _inputs():
    files = [os.path.join(CSRC, s) for s in SOURCES]
    files += [os.path.join(CSRC, h) for h in HEADERS if os.path.exists(os.path.join(CSRC, h))]
    files += [os.path.join(INCLUDE, "smem.h"), os.path.abspath(__file__)]
    return files


def _flavor(extra_flags=()) -> str:
    # what, besides the sources, decides the library's contents
    debug = os.environ.get("SMEM_DEBUG", "0") not in ("", "0")
    return " ".join(["debug" if debug else "release"] + list(extra_flags))


def up_to_date(extra_flags=()) -> bool:
    if not os.path.exists(LIB):
        return False
    try:
        with open(LIB + ".flavor") as f:
            if f.read().strip() != _flavor(extra_flags):
                return False  # built with other flags (e.g. the bounds-checking variant)
    except OSError:
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False, extra_flags=()) -> str:
    """SMEM_DEBUG=1 in the environment builds the bounds-checking variant
    (kernels check table, row and split indices and record an error instead
    of touching memory out of range)."""
    if not force and up_to_date(extra_flags):
        return LIB
    nvcc = _nvcc()
    os.makedirs(OBJ, exist_ok=True)
    common = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", f"-I{INCLUDE}", f"-I{CSRC}"] + list(extra_flags)
    if os.environ.get("SMEM_DEBUG", "0") not in ("", "0"):
        common.append("-DSMEM_DEBUG=1")

    def compile_one(src):
        out = os.path.join(OBJ, os.path.splitext(src)[0] + ".o")
        cmd = [nvcc, "-c", os.path.join(CSRC, src), "-o", out] + common
        if src.endswith(".cu"):
            cmd += ARCH + ["-Xptxas", "-v"] if verbose else ARCH
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return out, r.stderr

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose:
        for _, log in results:
            if log.strip():
                print(log)
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [nvcc, "-shared", "-o", tmp] + [o for o, _ in results] + ARCH + [
        "-cudart", "shared", "-Xlinker", f"-rpath,{_cuda_lib_dir(nvcc)}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(LIB + ".flavor", "w") as f:
        f.write(_flavor(extra_flags) + "\n")
    return LIB


if __name__ == "__main__":
    import sys

    print(build(force=True, verbose="-v" in sys.argv))
