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
import sysconfig

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libt2istore.so")
# CPython entry points for the per-request calls (csrc/pycall.c), linked
# against LIB
PYCALL_SRC = "pycall.c"
PYCALL = os.path.join(PKG, "_pycall" + (sysconfig.get_config_var("EXT_SUFFIX") or ".so"))

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
    files = [os.path.join(CSRC, f) for f in CXX_SOURCES + CU_SOURCES + HEADERS + [PYCALL_SRC]]
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


def _have_python_h() -> bool:
    return os.path.exists(os.path.join(sysconfig.get_paths()["include"], "Python.h"))


def is_stale() -> bool:
    outs = [LIB] + ([PYCALL] if _have_python_h() else [])
    if not all(os.path.exists(f) for f in outs):
        return True
    t = min(os.path.getmtime(f) for f in outs)
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
        log, _ = p.communicate()
        if verbose or ptxas_info or p.returncode:
            sys.stderr.write(log)
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
    if out is None:
        if _have_python_h():
            build_pycall(verbose)
        else:
            # the ctypes binding serves every call; only its per-call cost is higher
            sys.stderr.write("build: Python.h not found; the CPython binding (_pycall) is not built\n")
    return lib_path


def build_pycall(verbose: bool = False) -> str:
    """Compiles the CPython module of csrc/pycall.c next to LIB (linked
    against it, found through $ORIGIN). Raises on failure."""
    py_inc = sysconfig.get_paths()["include"]
    if not os.path.exists(os.path.join(py_inc, "Python.h")):
        raise RuntimeError(f"Python.h not found in {py_inc}: the CPython binding cannot be built")
    tmp = PYCALL + ".tmp"
    cmd = [os.environ.get("CC", "gcc"), "-O2", "-shared", "-fPIC", "-Wall", os.path.join(CSRC, PYCALL_SRC),
           "-I" + INCLUDE, "-I" + py_inc, "-L" + PKG, "-lt2istore", "-Wl,-rpath,$ORIGIN", "-o", tmp]
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if verbose or r.returncode:
        sys.stderr.write(r.stdout)
    if r.returncode:
        raise RuntimeError("CPython binding build failed: " + " ".join(cmd))
    os.replace(tmp, PYCALL)
    return PYCALL


def build_cdriver() -> str:
    """Compiles cdriver/handoff_step.c (the handoff workload driven from C
    through the C ABI) into _build/ against LIB and the CUDA runtime;
    returns the executable's path. Raises on failure."""
    cuda = _cuda_home()
    os.makedirs(BUILD, exist_ok=True)
    exe = os.path.join(BUILD, "handoff_step")
    lib64 = os.path.join(cuda, "lib64")
    cmd = [os.environ.get("CC", "gcc"), "-O2", "-std=c11", "-Wall", os.path.join(PKG, "cdriver", "handoff_step.c"),
           "-I" + INCLUDE, "-I" + os.path.join(cuda, "include"), "-L" + PKG, "-lt2istore", "-L" + lib64, "-lcudart",
           "-Wl,-rpath," + PKG + ":" + lib64, "-o", exe]
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode:
        raise RuntimeError("C driver build failed: " + " ".join(cmd) + "\n" + r.stdout)
    return exe


def ensure_built() -> str:
    """Builds the library if it is missing or older than its sources."""
    if is_stale():
        build()
    return LIB


if __name__ == "__main__":
    print(build(verbose=True, ptxas_info="--ptxas" in sys.argv))
