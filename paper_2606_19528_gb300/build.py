"""In-tree build of the CUDA library (sm_103a) and of the C input generator.

    python -m paper_2606_19528_gb300.build

compiles csrc/*.cu in parallel with nvcc into _lib/liblora_gb300.so and
synth_c/synth.c with gcc into synth_c/libsynth.so.  Outputs are rebuilt only
when a source or header is newer.
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "_lib", "liblora_gb300.so")
SYNTH_SRC = os.path.join(PKG, "synth_c", "synth.c")
SYNTH_LIB = os.path.join(PKG, "synth_c", "libsynth.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "--expt-relaxed-constexpr",
                     "-Xcompiler", "-fPIC,-O2", "-I", INCLUDE, "-I", CSRC]


def _nvcc() -> str:
    for c in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def _newer(out: str, deps) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(d) > t for d in deps)


def _run(cmd, verbose):
    if verbose:
        print(" ".join(cmd), flush=True)
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"command failed ({r.returncode}): {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    if verbose and (r.stdout or r.stderr):
        print(r.stdout + r.stderr, flush=True)
    return r


def build_synth(verbose: bool = False) -> str:
    if _newer(SYNTH_LIB, [SYNTH_SRC]):
        cc = shutil.which("gcc") or shutil.which("cc")
        _run([cc, "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC", "-shared",
              "-o", SYNTH_LIB, SYNTH_SRC, "-lm"], verbose)
    return SYNTH_LIB


def build_cuda(verbose: bool = False, ptxas_verbose: bool = False) -> str:
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    headers = sorted(glob.glob(os.path.join(CSRC, "*.h")) + glob.glob(os.path.join(CSRC, "*.cuh"))
                     + glob.glob(os.path.join(INCLUDE, "*.h")))
    os.makedirs(BUILD, exist_ok=True)
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    nvcc = _nvcc()
    objs = []
    jobs = []
    for s in srcs:
        o = os.path.join(BUILD, os.path.splitext(os.path.basename(s))[0] + ".o")
        objs.append(o)
        if _newer(o, [s] + headers) or ptxas_verbose:
            cmd = [nvcc] + NVCC_FLAGS + (["-Xptxas", "-v"] if ptxas_verbose else []) + ["-c", s, "-o", o]
            jobs.append(cmd)
    if jobs:
        with ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 4)) as ex:
            for r in ex.map(lambda c: _run(c, verbose or ptxas_verbose), jobs):
                pass
    if _newer(LIB, objs):
        cudalib = os.path.join(os.path.dirname(os.path.dirname(nvcc)), "lib64")
        _run([nvcc] + ARCH + ["-shared", "-cudart", "shared", "-o", LIB] + objs
             + ["-Xlinker", f"-rpath,{cudalib}"], verbose)
    return LIB


def build(verbose: bool = False) -> None:
    build_synth(verbose)
    build_cuda(verbose)


if __name__ == "__main__":
    build(verbose="-v" in sys.argv)
    if "--ptxas" in sys.argv:
        build_cuda(ptxas_verbose=True)
