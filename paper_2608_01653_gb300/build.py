"""In-tree build of libhatq.so for sm_103a (GB300) with nvcc.

Each translation unit is compiled in parallel with one -gencode
(arch=compute_103a, code=sm_103a), then linked into a shared library with the
CUDA runtime linked statically. The result lives in
paper_2608_01653_gb300/_build/ (git-ignored) and is rebuilt when a source or
header is newer than it.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "libhatq.so")
SOURCES = ["hatq_api.cu", "hatq_fwht.cu", "hatq_conv.cu", "hatq_conv_pieces.cu", "hatq_gdn.cu", "hatq_noalloc.cu",
           "hatq_profile.cu"]
HEADERS = [os.path.join(CSRC, "hatq_internal.h"), os.path.join(CSRC, "hatq_tc.h"), os.path.join(INCLUDE, "hatq.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libhatq")


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    files = [os.path.join(CSRC, s) for s in SOURCES] + HEADERS + [os.path.abspath(__file__)]
    return any(os.path.getmtime(f) > t for f in files)


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile libhatq.so if needed and return its path."""
    if not force and not _stale():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    flags = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-ffp-contract=off",
                    "-I", INCLUDE, "-I", CSRC]
    if verbose:
        flags += ["-Xptxas", "-v"]
    tag = str(os.getpid())

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.splitext(src)[0] + f".{tag}.o")
        cmd = [cc] + flags + ["-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose:
        for _, log in results:
            print(log)
    tmp = LIB + f".{tag}.tmp"
    cmd = [cc] + ARCH + ["-shared", "-o", tmp] + [o for o, _ in results]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link of libhatq.so failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    for o, _ in results:
        os.remove(o)
    return LIB


if __name__ == "__main__":
    import sys
    print(build(force=True, verbose="-v" in sys.argv))
