"""Build libmnmt.so (the sm_103a CUDA library behind include/mnmt.h), in-tree.

nvcc compiles each translation unit in parallel for sm_103a only, with
--fmad=false (every a*b+c of the method is two IEEE roundings unless a kernel
asks for a fused multiply-add explicitly) and host code with
-ffp-contract=off; the objects are linked into one shared library with the
static CUDA runtime.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libmnmt.so")
SOURCES = ["api.cu", "linear.cu", "linear_w4.cu", "gemm_tc.cu", "attention.cu", "rows.cu", "decode_cluster.cu",
           "noalloc.cu", "fakequant.cu"]
HEADERS = ["common.cuh", "epilogue.cuh", "internal.h", "mbarrier.cuh"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _nvcc():
    for cand in [os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"]:
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _flags(verbose_ptxas=False):
    f = ARCH + ["-O3", "-lineinfo", "-std=c++17", "--fmad=false", "-Xcompiler", "-fPIC,-ffp-contract=off",
                "-I", os.path.join(HERE, "..", "include")]
    if verbose_ptxas:
        f += ["-Xptxas", "-v"]
    return f


def _stale():
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    deps = [os.path.join(CSRC, s) for s in SOURCES + HEADERS] + [os.path.join(HERE, "..", "include", "mnmt.h")]
    return any(os.path.getmtime(p) > t for p in deps)


STAMPS_LIB = os.path.join(OUT_DIR, "libmnmt_stamps.so")


def build(force: bool = False, verbose_ptxas: bool = False, stamps: bool = False) -> str:
    """Build libmnmt.so; stamps=True builds the phase-timing debug variant
    libmnmt_stamps.so instead (the cluster decode step compiled with
    -DMNMT_DC_STAMPS; see phase_profile.py)."""
    lib = STAMPS_LIB if stamps else LIB
    if not force and not stamps and not _stale():
        return LIB
    os.makedirs(OUT_DIR, exist_ok=True)
    nvcc = _nvcc()
    flags = _flags(verbose_ptxas)

    def compile_one(src):
        obj = os.path.join(OUT_DIR, src.replace(".cu", ".stamps.o" if stamps else ".o"))
        extra = ["-DMNMT_DC_STAMPS"] if stamps and src == "decode_cluster.cu" else []
        cmd = [nvcc] + flags + extra + ["-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stderr}")
        return obj, r.stderr

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose_ptxas:
        for _, err in results:
            sys.stderr.write(err)
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [nvcc] + ARCH + ["-shared", "-o", tmp] + [o for o, _ in results]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose_ptxas="-v" in sys.argv, stamps="--stamps" in sys.argv))
