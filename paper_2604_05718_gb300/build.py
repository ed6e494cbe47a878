"""Builds libmpm.so (the C-ABI library) in-tree for sm_103a with nvcc.

Each .cu file under csrc/ is compiled in parallel to an object file in
_build/, then linked into paper_2604_05718_gb300/libmpm.so with the CUDA
runtime linked statically and only the mpm_* symbols exported.
"""

from __future__ import annotations

import concurrent.futures
import glob
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libmpm.so")
# The same sources with the device timeline compiled in (-DMPM_TRACE); see
# mpm_trace_read in include/mpm.h.  Used by `bench.py --timeline` only.
BUILD_TRACE = os.path.join(PKG, "_build_trace")
LIB_TRACE = os.path.join(PKG, "libmpm_trace.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden",
                     "-I", os.path.join(ROOT, "include"), "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the MPM library needs the CUDA toolkit to build")


def _headers() -> list:
    return glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(CSRC, "*.h")) + \
        [os.path.join(ROOT, "include", "mpm.h")]


def _stale(target: str, deps: list) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _run(cmd: list) -> None:
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"command failed ({res.returncode}): {' '.join(cmd)}\n{res.stdout}\n{res.stderr}")


def build(force: bool = False, extra_flags: list | None = None, trace: bool = False) -> str:
    """Compiles and links libmpm.so (libmpm_trace.so with trace=True) if any
    source changed; returns its path."""
    build_dir, lib_path = (BUILD_TRACE, LIB_TRACE) if trace else (BUILD, LIB)
    os.makedirs(build_dir, exist_ok=True)
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    headers = _headers()
    flags = NVCC_FLAGS + (["-DMPM_TRACE"] if trace else []) + list(extra_flags or [])
    jobs = []
    objs = []
    for src in srcs:
        obj = os.path.join(build_dir, os.path.basename(src)[:-3] + ".o")
        objs.append(obj)
        if force or _stale(obj, [src] + headers):
            jobs.append([nvcc(), "-c", src, "-o", obj] + flags)
    if jobs:
        with concurrent.futures.ThreadPoolExecutor(max_workers=min(8, len(jobs))) as ex:
            list(ex.map(_run, jobs))
    if force or jobs or _stale(lib_path, objs):
        tmp = lib_path + ".tmp"
        _run([nvcc(), "-shared", "-o", tmp] + objs + ARCH +
             ["-cudart", "static", "-Xlinker", "--version-script=" + os.path.join(CSRC, "exports.map")])
        os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    print(build(force=True))
