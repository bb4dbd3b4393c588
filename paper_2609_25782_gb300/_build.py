"""Compile libkvtier.so in-tree with nvcc for sm_103a.

The translation units (decode_kernels.cu, copy_kernels.cu, pool.cpp,
noalloc.cu) compile in parallel and are linked with the static CUDA runtime,
so the library needs only the driver at run time.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
LIB = os.path.join(HERE, "libkvtier.so")
SOURCES = ["decode_kernels.cu", "copy_kernels.cu", "pool.cpp", "noalloc.cu"]
HEADERS = ["kvt_internal.h", os.path.join("..", "..", "include", "kvtier.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libkvtier.so")


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    deps = [os.path.join(CSRC, s) for s in SOURCES + HEADERS] + [os.path.abspath(__file__)]
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale():
        return LIB
    cc = nvcc()
    out_dir = os.path.join(HERE, "_build")
    os.makedirs(out_dir, exist_ok=True)
    # KVT_EXTRA_NVCC_FLAGS: extra -D tuning definitions for experiments
    extra_flags = os.environ.get("KVT_EXTRA_NVCC_FLAGS", "").split()
    common = [cc, "-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", *ARCH,
              "-I", os.path.join(HERE, "..", "include"), *extra_flags]
    procs, objs = [], []
    for src in SOURCES:
        obj = os.path.join(out_dir, src + ".o")
        objs.append(obj)
        extra = ["-Xptxas", "-v"] if verbose and src.endswith(".cu") else []
        procs.append((src, subprocess.Popen(common + extra + ["-c", os.path.join(CSRC, src), "-o", obj],
                                            stdout=subprocess.PIPE, stderr=subprocess.STDOUT,
                                            text=True)))
    for src, p in procs:
        out, _ = p.communicate()
        if p.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{out}")
        if verbose and out:
            sys.stderr.write(out)
    tmp = LIB + ".tmp"
    res = subprocess.run([cc, "-shared", *ARCH, "-o", tmp, *objs], capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"link failed:\n{res.stdout}{res.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
