"""Compiles the CUDA sources into the in-tree C-ABI library liblitevlm_select.so.

sm_103a only (`-gencode arch=compute_103a,code=sm_103a`), translation units
compiled in parallel, static CUDA runtime, no link against libcuda (the driver
entry point for TMA descriptors is looked up at run time), so the library
loads on a machine without a GPU driver.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
from typing import List, Optional

PKG = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG, "csrc")
OBJ = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "liblitevlm_select.so")
# debug variant: NVTX ranges around every C-ABI call and the device / host
# mirror checks (LITEVLM_DEBUG); a separate library, loaded when LITEVLM_LIB
# names it
OBJ_DEBUG = os.path.join(PKG, "_build_debug")
LIB_DEBUG = os.path.join(PKG, "liblitevlm_select_debug.so")
SOURCES = ["api.cu", "score_tc.cu", "score_res.cu", "ctx_stats.cu", "topk.cu", "compact.cu", "splice.cu", "views.cu", "proj.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found")
    return path


def _compile(src: str, extra: List[str], objdir: str = OBJ) -> str:
    obj = os.path.join(objdir, os.path.splitext(src)[0] + ".o")
    cmd = [nvcc(), *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-c",
           os.path.join(CSRC, src), "-o", obj, *extra]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
    if r.stderr.strip():
        print(r.stderr.strip())
    return obj


def build(verbose_ptxas: bool = False, extra_flags: Optional[List[str]] = None, debug: bool = False) -> str:
    """Builds the library (or, with debug=True, the debug variant) and returns
    its path. LITEVLM_NVTX=1 in the environment adds the NVTX ranges to the
    release build too."""
    objdir, lib = (OBJ_DEBUG, LIB_DEBUG) if debug else (OBJ, LIB)
    os.makedirs(objdir, exist_ok=True)
    extra = list(extra_flags or [])
    if verbose_ptxas:
        extra += ["-Xptxas", "-v"]
    if debug:
        extra += ["-DLITEVLM_DEBUG", "-DLITEVLM_NVTX"]
    elif os.environ.get("LITEVLM_NVTX") == "1":
        extra += ["-DLITEVLM_NVTX"]
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra, objdir), SOURCES))
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [nvcc(), *ARCH, "-shared", "-o", tmp, *objs, "-ldl"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    import sys
    print(build(verbose_ptxas="-v" in sys.argv, debug="--debug" in sys.argv))
