"""Build libfastvr_attn.so in-tree with nvcc for sm_103a.

    python -m paper_2609_36757_gb300.build [--force]

Each translation unit compiles in parallel into _build/; the shared library is
linked next to this file with the CUDA runtime linked statically, so loading it
needs no CUDA driver (a host without a GPU can load it and list its symbols).
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libfastvr_attn.so")
# The debug variant: every computed global index of the append and attention
# kernels is checked before the access (FASTVR_BOUNDS_CHECK).
DEBUG_BUILD = os.path.join(HERE, "_build_debug")
DEBUG_LIB = os.path.join(HERE, "libfastvr_attn_debug.so")
INCLUDE = os.path.join(ROOT, "include")

SOURCES = ["fastvr_host.cpp", "kv_append.cu", "chunk_attn_fwd.cu",
           "chunk_attn_static.cu", "one_step.cu", "chunk_attn_bwd.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC",
         "-Xcompiler", "-fvisibility=hidden", "-I", INCLUDE, "-I", CSRC]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"),
                 "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build")


def _headers():
    hs = [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    hs += [os.path.join(CSRC, f) for f in os.listdir(CSRC)
           if f.endswith((".h", ".cuh"))]
    return hs


def _stale(target: str, deps) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _compile(nvcc: str, src: str, force: bool, extra, build_dir: str) -> str:
    obj = os.path.join(build_dir, os.path.splitext(src)[0] + ".o")
    path = os.path.join(CSRC, src)
    if force or _stale(obj, [path, __file__] + _headers()):
        cmd = [nvcc, "-c", path, "-o", obj] + ARCH + FLAGS + list(extra)
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if r.stderr.strip():
            sys.stderr.write(r.stderr)
    return obj


def _link(nvcc: str, lib: str, objs, force: bool) -> None:
    if force or _stale(lib, objs):
        cmd = [nvcc, "-shared", "-o", lib] + objs + ARCH + [
            "-cudart", "static", "-Xcompiler", "-fPIC"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")


def build(force: bool = False, verbose_ptxas: bool = False,
          debug: bool = True) -> str:
    """Build the release library (and, with debug, the index-checking one:
    both compile in one parallel pool).  Returns the release library path."""
    nvcc = _nvcc()
    extra = ["-Xptxas", "-v"] if verbose_ptxas else []
    jobs = [(s, extra, BUILD) for s in SOURCES]
    if debug:
        jobs += [(s, extra + ["-DFASTVR_BOUNDS_CHECK"], DEBUG_BUILD)
                 for s in SOURCES]
    for d in {j[2] for j in jobs}:
        os.makedirs(d, exist_ok=True)
    with cf.ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        objs = list(ex.map(lambda j: _compile(nvcc, j[0], force, j[1], j[2]),
                           jobs))
    _link(nvcc, LIB, objs[:len(SOURCES)], force)
    if debug:
        _link(nvcc, DEBUG_LIB, objs[len(SOURCES):], force)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv,
                verbose_ptxas="--ptxas-v" in sys.argv))
