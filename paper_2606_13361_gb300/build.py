"""In-tree build of libkvr.so for sm_103a (nvcc, no cmake).

Each translation unit compiles in its own nvcc process, in parallel; the
shared library links them with the static CUDA runtime.  Outputs land under
the package (git-ignored): _build/*.o and libkvr.so.
"""
from __future__ import annotations

import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libkvr.so")
SOURCES = ["kvr_api.cu", "kvr_attn.cu", "kvr_append.cu", "kvr_decode.cu", "kvr_artifact.cu", "kvr_layer.cu",
           "kvr_gemm.cu"]
HEADERS = [os.path.join(CSRC, h) for h in ("kvr_internal.h", "kvr_ptx.cuh", "kvr_rope.cuh", "kvr_artifact.cuh")] + [
    os.path.join(ROOT, "include", "kvr.h")]
NVCC_FLAGS = ["-std=c++17", "-O3", "-gencode", "arch=compute_103a,code=sm_103a", "-lineinfo",
              "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden"]


def _nvcc() -> str:
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def _stale(target: str, deps) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build_library(force: bool = False, verbose: bool = False, defines=(), extra_sources=(), build_dir: str = BUILD,
                  lib: str = LIB) -> str:
    """Compile and link the library.  `defines`, `extra_sources`, `build_dir`
    and `lib` serve variant builds (stage_trace.py); the defaults build
    libkvr.so."""
    os.makedirs(build_dir, exist_ok=True)
    nvcc = _nvcc()
    procs = []
    objs = []
    for src in list(SOURCES) + list(extra_sources):
        s = os.path.join(CSRC, src)
        o = os.path.join(build_dir, src.replace(".cu", ".o"))
        objs.append(o)
        if force or _stale(o, [s] + HEADERS):
            cmd = [nvcc] + NVCC_FLAGS + [f"-D{d}" for d in defines] + ["-c", s, "-o", o]
            if verbose:
                print(" ".join(cmd), file=sys.stderr)
            procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)))
    errors = []
    for src, p in procs:
        out, _ = p.communicate()
        if p.returncode != 0:
            errors.append(f"{src}:\n{out.decode(errors='replace')}")
        elif verbose and out:
            print(out.decode(errors="replace"), file=sys.stderr)
    if errors:
        raise RuntimeError("nvcc failed:\n" + "\n".join(errors))
    if force or _stale(lib, objs):
        tmp = lib + f".tmp{os.getpid()}"
        cuda_lib = os.path.join(os.path.dirname(os.path.dirname(_nvcc())), "lib64")
        cmd = [nvcc, "-shared", "-gencode", "arch=compute_103a,code=sm_103a", "-o", tmp] + objs + [
            "-L" + cuda_lib, "-Xlinker", "-rpath=" + cuda_lib]
        subprocess.check_call(cmd)
        os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose=True))
