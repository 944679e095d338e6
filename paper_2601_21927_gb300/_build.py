"""Builds libsonic.so (the CUDA kernels + C ABI) in-tree with nvcc for sm_103a.

Each .cu translation unit is compiled in parallel, then linked into
``paper_2601_21927_gb300/_lib/libsonic.so`` against the shared CUDA runtime
(the same libcudart torch loads).  A stamp of the sources and flags decides
whether a rebuild is needed.
"""
from __future__ import annotations

import hashlib
import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(HERE, "_lib")
LIB = os.path.join(OUT_DIR, "libsonic.so")

SOURCES = ["api.cu", "compact.cu", "decode.cu", "prefill.cu", "prefill_static.cu", "routed.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler",
              "-fvisibility=hidden", "--expt-relaxed-constexpr", "-I" + INCLUDE, "-I" + CSRC]


def _nvcc() -> str:
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: libsonic needs the CUDA 13 toolkit to build")
    return cand


def _stamp() -> str:
    h = hashlib.sha256()
    h.update(" ".join(ARCH + NVCC_FLAGS).encode())
    for d, names in ((CSRC, sorted(os.listdir(CSRC))), (INCLUDE, sorted(os.listdir(INCLUDE)))):
        for n in names:
            if n.endswith((".cu", ".cuh", ".h")):
                with open(os.path.join(d, n), "rb") as f:
                    h.update(n.encode())
                    h.update(f.read())
    return h.hexdigest()


def compile_library(lib_path: str, sources=SOURCES, defines=(), verbose: bool = False) -> str:
    """Compile `sources` (names under csrc/) with extra -D `defines` into the
    shared library `lib_path` (objects beside it); returns its path."""
    out_dir = os.path.dirname(os.path.abspath(lib_path))
    os.makedirs(out_dir, exist_ok=True)
    nvcc = _nvcc()
    tag = os.path.splitext(os.path.basename(lib_path))[0]

    def compile_one(src):
        obj = os.path.join(out_dir, f"{tag}_{src.replace('.cu', '.o')}")
        cmd = ([nvcc] + ARCH + NVCC_FLAGS + ["-D" + d for d in defines] +
               ["-c", os.path.join(CSRC, src), "-o", obj])
        if verbose:
            cmd += ["-Xptxas", "-v"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose:
            print(r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=len(sources)) as ex:
        objs = list(ex.map(compile_one, sources))
    tmp = lib_path + f".tmp{os.getpid()}"
    cmd = [nvcc] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib_path)
    return lib_path


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile libsonic.so if its sources changed; returns its path."""
    os.makedirs(OUT_DIR, exist_ok=True)
    stamp_path = os.path.join(OUT_DIR, "libsonic.stamp")
    stamp = _stamp()
    if (not force and os.path.exists(LIB) and os.path.exists(stamp_path)
            and open(stamp_path).read() == stamp):
        return LIB
    compile_library(LIB, SOURCES, verbose=verbose)
    with open(stamp_path, "w") as f:
        f.write(stamp)
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
