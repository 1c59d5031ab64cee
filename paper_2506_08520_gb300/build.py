"""Build ``libnystra.so`` (the C-ABI CUDA library) in-tree for sm_103a, and
``libnystra_host.so`` (the multi-core CPU path, ``host/nystra_host.c``).

Each ``csrc/*.cu`` translation unit is compiled in parallel with nvcc, then
linked into ``paper_2506_08520_gb300/libnystra.so``.  Objects go to
``paper_2506_08520_gb300/_build/`` (git-ignored).  Rebuilds only what changed.
The CPU library is plain C for the host's compiler defaults (no
machine-specific flags: the same source builds for x86-64 and Arm).
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libnystra.so")
HOST_SRC = os.path.join(PKG, "host", "nystra_host.c")
HOST_LIB = os.path.join(PKG, "libnystra_host.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "--expt-relaxed-constexpr", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-fvisibility=hidden", "-I", INCLUDE, "-I", CSRC]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _headers_mtime() -> float:
    hs = glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))
    return max((os.path.getmtime(h) for h in hs), default=0.0)


def _compile(src: str, extra: list[str]) -> str:
    obj = os.path.join(OUT_DIR, os.path.basename(src) + ".o")
    if os.path.exists(obj) and os.path.getmtime(obj) >= max(os.path.getmtime(src), _headers_mtime()):
        return obj
    cmd = [_nvcc(), *ARCH, *NVCC_FLAGS, *extra, "-c", src, "-o", obj + ".tmp"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stderr}")
    os.replace(obj + ".tmp", obj)
    return obj


def build(verbose: bool = False, extra: list[str] | None = None) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    with cf.ThreadPoolExecutor(max_workers=min(len(srcs), os.cpu_count() or 4)) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra or []), srcs))
    if os.path.exists(LIB) and os.path.getmtime(LIB) >= max(os.path.getmtime(o) for o in objs):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [_nvcc(), *ARCH, "-shared", "-cudart", "shared", "-o", tmp, *objs,
           "-Xlinker", "-rpath,/usr/local/cuda/lib64"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    os.replace(tmp, LIB)
    if verbose:
        print("built", LIB)
    return LIB


def build_host(verbose: bool = False) -> str:
    """Compile the multi-core CPU path into ``libnystra_host.so``."""
    deps = [HOST_SRC, os.path.join(INCLUDE, "nystra_host.h"), os.path.join(INCLUDE, "nystra.h"),
            os.path.abspath(__file__)]  # the flags below
    if os.path.exists(HOST_LIB) and os.path.getmtime(HOST_LIB) >= max(os.path.getmtime(f) for f in deps):
        return HOST_LIB
    tmp = HOST_LIB + f".tmp{os.getpid()}"
    # -fno-trapping-math lets the softmax loops' selects vectorise; -ffp-contract=fast
    # lets the compiler fuse multiply-adds where the ISA has them (strict -std=c11
    # turns that off).  No -ffast-math: the sums are not reassociated.
    cmd = [os.environ.get("CC", "gcc"), "-O3", "-std=c11", "-fopenmp", "-fno-math-errno", "-fno-trapping-math",
           "-ffp-contract=fast", "-fPIC", "-shared", "-fvisibility=hidden", "-I", INCLUDE, "-o", tmp, HOST_SRC, "-lm"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"host library build failed:\n{r.stderr}")
    os.replace(tmp, HOST_LIB)
    if verbose:
        print("built", HOST_LIB)
    return HOST_LIB


def ptxas_report(src: str) -> str:
    """Registers / spills / shared memory per kernel (``-Xptxas -v``) for one source file."""
    cmd = [_nvcc(), *ARCH, *NVCC_FLAGS, "-Xptxas", "-v", "-c", src, "-o", os.devnull]
    return subprocess.run(cmd, capture_output=True, text=True).stderr


if __name__ == "__main__":
    if "--ptxas" in sys.argv:
        for s in sorted(glob.glob(os.path.join(CSRC, "*.cu"))):
            print(ptxas_report(s))
    else:
        build(verbose=True)
        build_host(verbose=True)
