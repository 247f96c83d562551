"""Build libdarb.so (and libdarb_baselines.so) in-tree with nvcc for sm_103a (GB300).

Each CUDA translation unit compiles in parallel to an object under ``_build/``
and the objects link into ``paper_1911_08020_gb300/libdarb.so``, which exports
only the C ABI declared in ``include/darb.h``.  ``libdarb_baselines.so`` holds
the cuSPARSE comparison products of ``include/darb_baselines.h``; it is a
separate library so that libdarb never links the vendor sparse library.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libdarb.so")
BASE_LIB = os.path.join(PKG, "libdarb_baselines.so")
BASE_SOURCES = ["baselines.cu"]
SOURCES = ["darb_api.cu", "assign.cu", "encode.cu", "spmm.cu", "spmm_batch.cu", "spmm_tc.cu", "rnn.cu", "rnn_batch.cu",
           "noalloc.cu", "sequence.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libdarb")


def _inputs():
    files = [os.path.join(CSRC, s) for s in SOURCES + BASE_SOURCES]
    files += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    files += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h")]
    files += [os.path.abspath(__file__)]
    return files


def up_to_date() -> bool:
    if not os.path.exists(LIB) or not os.path.exists(BASE_LIB):
        return False
    t = min(os.path.getmtime(LIB), os.path.getmtime(BASE_LIB))
    return all(os.path.getmtime(f) <= t for f in _inputs())


def _cuda_lib_dir() -> str:
    return os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(nvcc()))), "lib64")


def _link(objs, out, extra=()):
    tmp = out + f".tmp{os.getpid()}"
    cmd = [nvcc(), "-shared", *objs, "-o", tmp, *ARCH, "-Xcompiler", "-fPIC", *extra]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link of {os.path.basename(out)} failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out)


def _compile(src: str, ptxas_verbose: bool) -> str:
    obj = os.path.join(BUILD, os.path.splitext(src)[0] + ".o")
    cmd = [nvcc(), "-c", os.path.join(CSRC, src), "-o", obj, "-O3", "-std=c++17", *ARCH,
           "-lineinfo", "-Xcompiler", "-fPIC,-fvisibility=hidden", "-I", INCLUDE, "-I", CSRC,
           "-DDARB_BUILDING_LIBRARY"]
    if ptxas_verbose:
        cmd += ["-Xptxas", "-v"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
    if ptxas_verbose:
        sys.stderr.write(r.stderr)
    return obj


def build(force: bool = False, ptxas_verbose: bool = False) -> str:
    """Compile and link libdarb.so if any input changed (or `force`); returns its path."""
    if not force and not ptxas_verbose and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    srcs = SOURCES + BASE_SOURCES
    with cf.ThreadPoolExecutor(max_workers=len(srcs)) as ex:
        objs = dict(zip(srcs, ex.map(lambda s: _compile(s, ptxas_verbose), srcs)))
    _link([objs[s] for s in SOURCES], LIB, ["-ldl"])   # NVTX loads a profiler's injection library
    libdir = _cuda_lib_dir()
    _link([objs[s] for s in BASE_SOURCES], BASE_LIB, ["-L" + libdir, "-lcusparse", "-Xlinker", "-rpath=" + libdir])
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, ptxas_verbose="-v" in sys.argv))
