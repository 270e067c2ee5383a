"""Builds ``lib/libpipo.so`` (the C-ABI library) for sm_103a with nvcc: the
host code and the kernel families are separate translation units, compiled
in parallel and linked into one shared library."""
from __future__ import annotations

import concurrent.futures
import hashlib
import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIBDIR = os.path.join(PKG, "lib")
LIB = os.path.join(LIBDIR, "libpipo.so")
# the host code first (the longest units start first)
SOURCES = ["k_gemv_bf16.cu", "k_gemv_f32.cu", "k_attn.cu", "pipo_capi.cu", "k_tc.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _digest() -> str:
    h = hashlib.sha256()
    for d in (CSRC, INCLUDE):
        for name in sorted(os.listdir(d)):
            p = os.path.join(d, name)
            if os.path.isfile(p):
                h.update(name.encode())
                with open(p, "rb") as f:
                    h.update(f.read())
    h.update(" ".join(ARCH + extra_flags()).encode())
    return h.hexdigest()


def extra_flags() -> list:
    """Experiment flags for every unit, e.g. PIPO_NVCC_FLAGS="-DPIPO_STREAM_THREADS=384
    -DPIPO_STREAM_CTAS_PER_SM=2" (the build-time switches of the kernels)."""
    return os.environ.get("PIPO_NVCC_FLAGS", "").split()


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if c and (os.path.isabs(c) and os.path.exists(c) or not os.path.isabs(c)):
            return c
    return "nvcc"


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile the library if its sources changed; returns its path."""
    os.makedirs(LIBDIR, exist_ok=True)
    stamp = LIB + ".sha256"
    dig = _digest()
    if not force and os.path.exists(LIB) and os.path.exists(stamp) and open(stamp).read() == dig:
        return LIB
    tag = f".tmp{os.getpid()}"
    flags = ["-O3", "-std=c++17", "-lineinfo", *ARCH, "-Xcompiler", "-fPIC,-fvisibility=hidden",
             "-I", INCLUDE, "-I", CSRC] + extra_flags() + (["-Xptxas=-v"] if verbose else [])

    def compile_unit(src: str) -> str:
        obj = os.path.join(LIBDIR, os.path.splitext(src)[0] + tag + ".o")
        cmd = [nvcc(), *flags, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            print(" ".join(cmd), file=sys.stderr)
        subprocess.check_call(cmd)
        return obj

    with concurrent.futures.ThreadPoolExecutor(max_workers=min(len(SOURCES), os.cpu_count() or 1)) as pool:
        objs = list(pool.map(compile_unit, SOURCES))
    tmp = LIB + tag
    try:
        subprocess.check_call([nvcc(), *ARCH, "-shared", "-o", tmp, *objs])
    finally:
        for o in objs:
            if os.path.exists(o):
                os.remove(o)
    os.replace(tmp, LIB)
    with open(stamp, "w") as f:
        f.write(dig)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
