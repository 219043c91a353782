"""Builds the SCM library (libtrident_scm.so) in-tree with nvcc for sm_103a.

One translation unit per kernel family plus the host core, compiled in parallel and
linked into one shared object with the CUDA runtime linked statically, so that the
library loads on machines without a GPU driver (it reaches the driver at run time)."""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INC = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIBDIR = os.path.join(PKG, "_lib")
LIB = os.path.join(LIBDIR, "libtrident_scm.so")
SOURCES = ["scm.cpp", "tree.cpp", "addnorm.cu", "rmsnorm.cu", "rope.cu", "swiglu.cu", "pointwise.cu", "chain.cu",
           "noalloc.cu"]
HEADERS = ["internal.h", "device_common.cuh", "tree.h", "measure.h"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden",
         "-I", INC, "-I", CSRC]


def nvcc():
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def _stale(target, deps):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force=False, verbose=False, extra_flags=()):
    os.makedirs(BUILD, exist_ok=True)
    os.makedirs(LIBDIR, exist_ok=True)
    hdrs = [os.path.join(CSRC, h) for h in HEADERS] + [os.path.join(INC, "trident_scm.h")]
    objs, jobs = [], []
    for src in SOURCES:
        s = os.path.join(CSRC, src)
        o = os.path.join(BUILD, src + ".o")
        objs.append(o)
        if force or _stale(o, [s] + hdrs):
            jobs.append([nvcc(), *ARCH, *FLAGS, *extra_flags, "-c", s, "-o", o])

    def run(cmd):
        if verbose:
            print(" ".join(cmd), file=sys.stderr)
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed:\n" + " ".join(cmd) + "\n" + r.stdout + r.stderr)
        return r.stdout + r.stderr

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        for out in ex.map(run, jobs):
            if verbose and out.strip():
                print(out, file=sys.stderr)
    if force or jobs or _stale(LIB, objs):
        run([nvcc(), *ARCH, "-shared", "-o", LIB + ".tmp", *objs])
        os.replace(LIB + ".tmp", LIB)
    build_fastcall(force, verbose)
    return LIB


def build_fastcall(force=False, verbose=False):
    """The CPython fast-call shim of the binding (linked against the library; built only
    where the Python headers are installed -- the binding uses ctypes otherwise)."""
    import sysconfig
    inc = sysconfig.get_paths()["include"]
    if not os.path.exists(os.path.join(inc, "Python.h")):
        return None
    src = os.path.join(CSRC, "fastcall.c")
    out = os.path.join(PKG, "_fastcall" + sysconfig.get_config_var("EXT_SUFFIX"))
    if not force and not _stale(out, [src, LIB, os.path.join(INC, "trident_scm.h")]):
        return out
    cmd = ["gcc", "-O2", "-shared", "-fPIC", "-I", inc, "-I", INC, src, "-o", out + ".tmp",
           "-L", LIBDIR, "-ltrident_scm", "-Wl,-rpath,$ORIGIN/_lib"]
    if verbose:
        print(" ".join(cmd), file=sys.stderr)
    subprocess.run(cmd, check=True)
    os.replace(out + ".tmp", out)
    return out


if __name__ == "__main__":
    flags = (["-Xptxas", "-v"] if "--ptxas" in sys.argv else []) + (["-DTRIDENT_NVTX"] if "--nvtx" in sys.argv else [])
    # --nvtx: NVTX ranges around the boundary calls (off by default); rebuild without it to
    # remove them again (--force)
    print(build(force="--force" in sys.argv or "--nvtx" in sys.argv, verbose=True, extra_flags=flags))
