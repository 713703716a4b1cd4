"""Build the CUDA library in-tree: nvcc for sm_103a, one -gencode, the
translation units compiled in parallel, then linked into libmixattn.so next to
this file (shared cudart, so the process shares one CUDA runtime with torch)."""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(HERE, "libmixattn.so")
SOURCES = ["mx_api.cpp", "mx_layer.cu", "mx_noalloc.cu", "mx_ops.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
         "-I", os.path.join(ROOT, "include")]


def _nvcc():
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def _compile(src, extra=()):
    obj = os.path.join(BUILD, os.path.basename(src) + ".o")
    cmd = [_nvcc(), *ARCH, *FLAGS, *extra, "-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    return obj, r.stderr


def build_library(verbose: bool = False) -> str:
    os.makedirs(BUILD, exist_ok=True)
    srcs = [os.path.join(CSRC, s) for s in SOURCES]
    with ThreadPoolExecutor(len(srcs)) as ex:
        res = list(ex.map(lambda s: _compile(s, ["-Xptxas", "-v"] if verbose else []), srcs))
    if verbose:
        for _, log in res:
            sys.stderr.write(log)
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [_nvcc(), *ARCH, "-shared", "-cudart", "shared", "-o", tmp] + [o for o, _ in res] + ["-lcublas"]
    subprocess.check_call(cmd)
    os.replace(tmp, LIB)
    return LIB


def build_synth() -> str:
    """The seeded input generator's device fill (test/bench support)."""
    src = os.path.join(ROOT, "synth", "fill.cu")
    out = os.path.join(ROOT, "synth", "libsynth.so")
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call([_nvcc(), *ARCH, "-O3", "-std=c++17", "-Xcompiler", "-fPIC",
                           "-shared", "-cudart", "shared", src, "-o", tmp])
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build_library(verbose="-v" in sys.argv))
