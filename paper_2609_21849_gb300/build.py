"""Builds libqlin.so in-tree for sm_103a with nvcc (no cmake, no torch
extension machinery): each .cu file is compiled in parallel, then linked with
the static CUDA runtime into ``paper_2609_21849_gb300/_lib/libqlin.so``."""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB_DIR = os.path.join(HERE, "_lib")
LIB = os.path.join(LIB_DIR, "libqlin.so")
SOURCES = ["qlin_api.cu", "qlin_quant.cu", "qlin_gemm.cu"]
# the tensor-core rate probe of the measurement harness: a library of its own
PROBE_LIB = os.path.join(LIB_DIR, "libqlin_probe.so")
PROBE_SOURCES = ["qlin_probe.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _flags():
    # QLIN_BUILD_DEFINES: extra -D options (the kernels' build-time layout
    # choices, e.g. "-DQLIN_WIDE_NVFP4=0"); empty for the default build
    extra = os.environ.get("QLIN_BUILD_DEFINES", "").split()
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                   "-I" + INCLUDE, "-I" + CSRC] + extra


def _inputs():
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    deps += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    return deps


def _fresh(lib):
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(d) <= t for d in _inputs())


def build(force: bool = False, verbose: bool = False) -> str:
    """Build libqlin.so and libqlin_probe.so (all translation units compiled
    in parallel); returns the path of libqlin.so."""
    os.makedirs(LIB_DIR, exist_ok=True)
    if not force and _fresh(LIB) and _fresh(PROBE_LIB):
        return LIB
    cc = nvcc()

    def compile_one(src):
        obj = os.path.join(LIB_DIR, src.replace(".cu", ".o"))
        cmd = [cc] + _flags() + ["-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        if verbose:
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    srcs = SOURCES + PROBE_SOURCES
    with cf.ThreadPoolExecutor(len(srcs)) as ex:
        objs = dict(zip(srcs, ex.map(compile_one, srcs)))
    for lib, group in ((LIB, SOURCES), (PROBE_LIB, PROBE_SOURCES)):
        tmp = lib + ".tmp"
        cmd = ([cc] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + [objs[f] for f in group]
               + ["-ldl", "-lpthread", "-lrt"])
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
