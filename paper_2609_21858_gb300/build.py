"""Build libpps.so (sm_103a) in-tree with nvcc: one process per translation
unit, then one link.  Used by ``__graft_entry__.build()``; run directly with
``python -m paper_2609_21858_gb300.build``."""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
OUT = os.path.join(PKG, "_lib")
LIB = os.path.join(OUT, "libpps.so")
SOURCES = ["pps_race.cu", "pps_misc.cu", "pps_api.cu"]
HEADERS = ["pps_device.cuh", "pps_internal.h", "pps_trunc.cuh", "pps_lmhead.cuh"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if c and (os.path.sep not in c or os.path.exists(c)):
            return c
    return "nvcc"


def _stale(target: str, deps) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


# Library variants: the default (Philox4x32-10) and the cheaper keyed source
# (Philox4x32-7), each from the same sources with its own objects.
VARIANTS = {"": [], "_r7": ["-DPPS_PHILOX_ROUNDS=7"]}


def lib_path(variant: str = "") -> str:
    return os.path.join(OUT, f"libpps{variant}.so")


def build(force: bool = False, verbose: bool = False) -> str:
    os.makedirs(OUT, exist_ok=True)
    hdrs = [os.path.join(CSRC, h) for h in HEADERS] + [os.path.join(ROOT, "include", "pps.h")]
    flags = ["-std=c++17", "-O3", "-lineinfo", "-Xcompiler", "-fPIC", "-I" + os.path.join(ROOT, "include")] + ARCH
    flags += os.environ.get("PPS_NVCC_FLAGS", "").split()  # extra flags for experiments (e.g. -DPPS_RACE_MIN_BLOCKS=4)

    def compile_one(job):
        variant, src = job
        s = os.path.join(CSRC, src)
        d = os.path.join(OUT, "obj" + variant)
        os.makedirs(d, exist_ok=True)
        o = os.path.join(d, src.replace(".cu", ".o"))
        if force or _stale(o, [s] + hdrs):
            cmd = [nvcc()] + flags + VARIANTS[variant] + ["-c", s, "-o", o]
            if verbose:
                print(" ".join(cmd), flush=True)
            subprocess.run(cmd, check=True)
        return o

    jobs = [(v, src) for v in VARIANTS for src in SOURCES]
    with ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        objs = list(ex.map(compile_one, jobs))
    for i, v in enumerate(VARIANTS):
        vobjs = objs[i * len(SOURCES):(i + 1) * len(SOURCES)]
        target = lib_path(v)
        if force or _stale(target, vobjs):
            tmp = target + f".tmp{os.getpid()}"
            cmd = [nvcc()] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + vobjs
            if verbose:
                print(" ".join(cmd), flush=True)
            subprocess.run(cmd, check=True)
            os.replace(tmp, target)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
