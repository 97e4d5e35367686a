"""Builds the CUDA library ``libgrpo_gb300.so`` in-tree with nvcc for sm_103a.

Each translation unit is compiled in parallel to an object file under ``_build/``, then the
objects are linked into a shared library next to this file (CUDA runtime linked statically, the
driver's TMA encoder fetched at run time, so only ``libcuda`` from the driver is needed).

Compile-time tuning knobs of the GEMM kernels can be overridden with the environment variable
``GRPO_DEFINES`` (comma-separated NAME=VALUE, each passed as -DGRPO_NAME=VALUE), e.g.
``GRPO_DEFINES=FWD_TILES_PER_STRIP=8,GROUP_M_DH=16``: ``FWD_TILES_PER_STRIP`` (vocabulary tiles
merged per forward work unit) and ``GROUP_M_FWD`` / ``GROUP_M_DZ`` / ``GROUP_M_DH`` /
``GROUP_M_DW`` (raster groups, in 128-row tiles). Objects are rebuilt whenever the value changes.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libgrpo_gb300.so")
SOURCES = ["api.cu", "gemm_tc.cu", "small_kernels.cu", "fwd_static_scratch.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libgrpo_gb300.so")


def _stale(obj: str, deps) -> bool:
    if not os.path.exists(obj):
        return True
    t = os.path.getmtime(obj)
    return any(os.path.getmtime(d) > t for d in deps)


def defines() -> list:
    """-D flags from GRPO_DEFINES (see the module docstring)."""
    spec = os.environ.get("GRPO_DEFINES", "").strip()
    out = []
    for item in filter(None, (x.strip() for x in spec.split(","))):
        name, _, value = item.partition("=")
        if not name.isidentifier() or not value.lstrip("-").isdigit():
            raise ValueError(f"GRPO_DEFINES: bad item {item!r} (want NAME=integer)")
        out.append(f"-DGRPO_{name}={value}")
    return out


def build(verbose: bool = False, ptxas_info: bool = False) -> str:
    os.makedirs(BUILD, exist_ok=True)
    headers = [os.path.join(CSRC, h) for h in os.listdir(CSRC) if h.endswith((".h", ".cuh"))]
    headers.append(os.path.join(os.path.dirname(HERE), "include", "grpo.h"))
    cc = nvcc()
    extra = (["-Xptxas", "-v"] if ptxas_info else []) + defines()
    # objects remember the defines they were built with: a change rebuilds them
    stamp = os.path.join(BUILD, "defines.txt")
    if not os.path.exists(stamp) or open(stamp).read() != " ".join(defines()):
        for f in os.listdir(BUILD):
            if f.endswith(".o"):
                os.remove(os.path.join(BUILD, f))
        with open(stamp, "w") as fh:
            fh.write(" ".join(defines()))

    def compile_one(src):
        s = os.path.join(CSRC, src)
        o = os.path.join(BUILD, src.replace(".cu", ".o"))
        if not (ptxas_info or _stale(o, [s, *headers])):
            return o, ""
        cmd = [cc, *ARCH, *FLAGS, *extra, "-c", s, "-o", o]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        return o, r.stdout + r.stderr

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    objs = [o for o, _ in results]
    if verbose or ptxas_info:
        for _, log in results:
            if log:
                print(log, file=sys.stderr)
    if _stale(LIB, objs):
        cmd = [cc, *ARCH, "-shared", "-o", LIB, *objs]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc link failed:\n{r.stdout}\n{r.stderr}")
    return LIB


if __name__ == "__main__":
    print(build(verbose=True, ptxas_info="--ptxas" in sys.argv))
