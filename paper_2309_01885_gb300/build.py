"""Builds libqe.so (the CUDA kernels and the C ABI of include/qe.h) in-tree.

    python -m paper_2309_01885_gb300.build        # or build_lib() from Python

Each translation unit is compiled by its own nvcc process (in parallel, the
slowest first) for sm_103a only, then linked into paper_2309_01885_gb300/_build/libqe.so with the
static CUDA runtime.  The driver API is reached through
cudaGetDriverEntryPointByVersion, so the library has no link-time dependency on
libcuda and loads on machines without a GPU driver.
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
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(OUT_DIR, "libqe.so")
# the sweep kernels' instantiations are spread over the qe_sweep_*.cu units (one
# kernel family and block width each) so that no single unit holds up the build
SOURCES = ["qe_sweep_seq256.cu", "qe_sweep_chg256.cu", "qe_sweep_rows256.cu", "qe_sweep_seq256r.cu",
           "qe_sweep_chg.cu", "qe_sweep_rows.cu", "qe_sweep_seq.cu", "qe_gemm.cu", "qe_api.cu", "qe_cd.cu",
           "qe_outlier.cu", "qe_noalloc.cu", "qe_stream.cu", "qe_pack.cu", "qe_select.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
              f"-I{os.path.join(ROOT, 'include')}", f"-I{CSRC}"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libqe")


def _deps_mtime() -> float:
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    files.append(os.path.join(ROOT, "include", "qe.h"))
    files.append(os.path.abspath(__file__))
    return max(os.path.getmtime(f) for f in files)


def build_lib(force: bool = False, verbose: bool = False) -> str:
    """Compile and link libqe.so; returns its path.  Skips work when up to date."""
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= _deps_mtime():
        return LIB
    os.makedirs(OUT_DIR, exist_ok=True)
    nvcc = _nvcc()

    def compile_one(src: str) -> str:
        obj = os.path.join(OUT_DIR, src.replace(".cu", ".o"))
        cmd = [nvcc, *ARCH, *NVCC_FLAGS, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{res.stdout}\n{res.stderr}")
        return obj

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"link failed:\n{res.stdout}\n{res.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build_lib(force="--force" in sys.argv, verbose=True))
