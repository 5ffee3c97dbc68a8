"""Build libdopr.so in-tree with nvcc for sm_103a.

Each .cu translation unit compiles in parallel to an object file under
``_build/``; the objects link into ``_build/libdopr.so`` (static CUDA runtime,
no libcuda link: the driver's tensor-map encoder is resolved at run time).
Objects are rebuilt when their source or any header is newer.

``build(checked=True)`` makes the checked variant under ``_build_checked/``
(compiled with -DDOPR_CHECKED): every data-dependent index into a global
buffer is tested against the buffer's extent, and a failed test skips the
access and makes the call return DOPR_ERR_INTERNAL.  It stands in for a
memory checker; the binding loads it when DOPR_CHECKED=1 is set.
"""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD, "libdopr.so")
BUILD_CHECKED = os.path.join(HERE, "_build_checked")
LIB_CHECKED = os.path.join(BUILD_CHECKED, "libdopr.so")
SOURCES = ["abi.cu", "k_gemm.cu", "k_attn.cu", "k_attn_tc.cu", "k_select.cu", "k_rows.cu", "k_pack.cu", "k_pack_noalloc.cu"]
HEADERS = [os.path.join(CSRC, "device_common.cuh"), os.path.join(CSRC, "internal.h"),
           os.path.join(ROOT, "include", "dopr.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
                     "-I", os.path.join(ROOT, "include"), "-Xptxas", "-warn-spills"]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.sep not in cand or os.path.exists(cand)):
            return cand
    return "nvcc"


def _stale(out: str, deps) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(d) > t for d in deps)


def _compile(src: str, verbose: bool, checked: bool = False) -> str:
    path = os.path.join(CSRC, src)
    obj = os.path.join(BUILD_CHECKED if checked else BUILD, src.replace(".cu", ".o"))
    if _stale(obj, [path] + HEADERS):
        cmd = [_nvcc()] + NVCC_FLAGS + (["-DDOPR_CHECKED"] if checked else []) + ["-c", path, "-o", obj + ".tmp"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        os.replace(obj + ".tmp", obj)
    return obj


def build(verbose: bool = False, checked: bool = False) -> str:
    """Compile and link libdopr.so (the checked variant when `checked`); returns its path."""
    out_dir, lib = (BUILD_CHECKED, LIB_CHECKED) if checked else (BUILD, LIB)
    os.makedirs(out_dir, exist_ok=True)
    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, verbose, checked), SOURCES))
    if _stale(lib, objs):
        cmd = [_nvcc()] + ARCH + ["-shared", "-o", lib + ".tmp"] + objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(lib + ".tmp", lib)
    return lib


if __name__ == "__main__":
    print(build(verbose=True, checked="--checked" in sys.argv[1:]))
