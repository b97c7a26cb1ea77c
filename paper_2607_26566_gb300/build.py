"""Builds libt2istore.so in-tree for sm_103a (GB300).

Host control (C++17, g++) and the store with its CUDA kernels (nvcc, one
-gencode for compute_103a/sm_103a) are compiled in parallel and linked into
one shared library next to this file. The CUDA runtime is linked statically
and the driver API is reached through the runtime, so the library loads on a
machine without a GPU driver (only the t2i_ctl_* calls work there).
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libt2istore.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CXX_SOURCES = ["control.cpp", "ctl_capi.cpp", "prefix.cpp"]
CU_SOURCES = ["store.cu"]
HEADERS = ["control.hpp", "common.hpp", "deps.hpp", "kernels.cuh", "launch.cuh", "exports.map"]


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH") or "/usr/local/cuda"
    if not os.path.exists(os.path.join(home, "bin", "nvcc")):
        nvcc = shutil.which("nvcc")
        if nvcc:
            home = os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return home


def _inputs() -> list[str]:
    files = [os.path.join(CSRC, f) for f in CXX_SOURCES + CU_SOURCES + HEADERS]
    return files + [os.path.join(INCLUDE, "t2istore.h"), os.path.abspath(__file__)]


def kernel_source_hash() -> str:
    """Short hash of the device code and the launch packing (ties profiles to
    what a launch does)."""
    import hashlib

    h = hashlib.sha256()
    for f in ("kernels.cuh", "launch.cuh"):
        with open(os.path.join(CSRC, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:12]


def is_stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(f) > t for f in _inputs())


def build(verbose: bool = False, ptxas_info: bool = False, defines=(), out: str | None = None,
          build_dir: str | None = None) -> str:
    """Compiles and links the library; returns its path. Raises on failure.
    ``defines`` (e.g. ["T2I_TUNE_VEC=8"]) and ``out`` build a variant of the
    kernels' launch shape elsewhere (tuning sweeps)."""
    lib_path = out or LIB
    bdir = build_dir or BUILD
    os.makedirs(bdir, exist_ok=True)
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    inc = ["-I" + INCLUDE, "-I" + CSRC, "-I" + os.path.join(cuda, "include")]
    jobs = []
    for f in CXX_SOURCES:
        obj = os.path.join(bdir, f + ".o")
        jobs.append(([os.environ.get("CXX", "g++"), "-O2", "-std=c++17", "-fPIC", "-Wall", "-ffp-contract=off", "-c",
                      os.path.join(CSRC, f), "-o", obj] + inc, obj))
    for f in CU_SOURCES:
        obj = os.path.join(bdir, f + ".o")
        cmd = [nvcc, "-O3", "-std=c++17", *ARCH, "-lineinfo", "-Xcompiler", "-fPIC,-Wall",
               "-c", os.path.join(CSRC, f), "-o", obj] + inc + ["-D" + d for d in defines]
        if ptxas_info:
            cmd += ["-Xptxas", "-v"]
        jobs.append((cmd, obj))
    procs = [(subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True), cmd, obj)
             for cmd, obj in jobs]
    objs = []
    errors = []
    for p, cmd, obj in procs:
        out, _ = p.communicate()
        if verbose or ptxas_info or p.returncode:
            sys.stderr.write(out)
        if p.returncode:
            errors.append(" ".join(cmd))
        objs.append(obj)
    if errors:
        raise RuntimeError("compilation failed:\n" + "\n".join(errors))
    tmp = lib_path + ".tmp"
    link = [nvcc, "-shared", *ARCH, "-o", tmp, *objs, "-cudart", "static", "-lpthread", "-ldl",
            "-Xlinker", "--version-script=" + os.path.join(CSRC, "exports.map")]
    r = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if verbose or r.returncode:
        sys.stderr.write(r.stdout)
    if r.returncode:
        raise RuntimeError("link failed: " + " ".join(link))
    os.replace(tmp, lib_path)
    return lib_path


def ensure_built() -> str:
    """Builds the library if it is missing or older than its sources."""
    if is_stale():
        build()
    return LIB


if __name__ == "__main__":
    print(build(verbose=True, ptxas_info="--ptxas" in sys.argv))
