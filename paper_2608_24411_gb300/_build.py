"""In-tree build of the CUDA library ``_lib/libresispec.so`` for sm_103a."""
from __future__ import annotations

import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
LIBDIR = os.path.join(HERE, "_lib")
LIB = os.path.join(LIBDIR, "libresispec.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "resispec.h")
UNITS = ("resispec.cu", "kern_resident_f32.cu", "kern_resident_bf16.cu", "kern_stream_f32.cu",
         "kern_stream_bf16.cu", "kern_stream_var_f32.cu", "kern_stream_var_bf16.cu")
SOURCES = [os.path.join(CSRC, f) for f in UNITS + ("kernels.h", "verify_kernel.cuh",
                                                   "verify_stream.cuh", "specinfer.cuh",
                                                   "dfloat.cuh", "philox.cuh", "ptx.cuh")]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.sep not in cand or os.path.exists(cand)):
            return cand
    return "nvcc"


def stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in SOURCES + [HEADER])


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile the library (nvcc, -gencode arch=compute_103a,code=sm_103a): one
    object per translation unit, compiled in parallel, then one shared link."""
    if not force and not stale():
        return LIB
    os.makedirs(LIBDIR, exist_ok=True)
    tag = f".tmp{os.getpid()}"
    flags = [nvcc(), "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo",
             "-std=c++17", "-Xcompiler", "-fPIC"]
    if verbose:
        flags.append("-Xptxas=-v")
    objs, procs = [], []
    for u in UNITS:
        obj = os.path.join(LIBDIR, os.path.splitext(u)[0] + tag + ".o")
        objs.append(obj)
        procs.append(subprocess.Popen(flags + ["-c", "-o", obj, os.path.join(CSRC, u)]))
    failed = [u for u, p in zip(UNITS, procs) if p.wait() != 0]
    try:
        if failed:
            raise subprocess.CalledProcessError(1, f"nvcc {' '.join(failed)}")
        tmp = LIB + tag
        subprocess.run([nvcc(), "-gencode", "arch=compute_103a,code=sm_103a", "-shared", "-o",
                        tmp] + objs, check=True)
        os.replace(tmp, LIB)
    finally:
        for o in objs:
            if os.path.exists(o):
                os.remove(o)
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
