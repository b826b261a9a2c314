"""Builds libsphq.so, the sm_103a CUDA library behind include/sphq.h, and
libsphq_study.so, the benchmark's 16-D gather-rate study (not part of the C ABI).

Plain nvcc, one translation unit per source compiled in parallel, static CUDA
runtime, no cmake.  The output lands next to this file (in-tree) and is
git-ignored; it must be rebuilt on each machine (the GPU machine is aarch64).
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libsphq.so")
SOURCES = ["sphq_api.cu", "sphq_gemv.cu", "sphq_gemv_splits.cu", "sphq_gemm.cu",
           "sphq_encode.cu", "sphq_io.cu", "sphq_noalloc.cu", "sphq_codebook.cu",
           "sphq_dim16.cu"]
STUDY_SRC = os.path.join(CSRC, "study", "gather16.cu")
STUDY_LIB = os.path.join(HERE, "libsphq_study.so")
HEADERS = ["sphq_layout.cuh", "sphq_gemv_kernel.cuh", "sphq_umma.cuh", "sphq_internal.h"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xptxas", "-v",
         "--expt-relaxed-constexpr"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _inputs():
    hdr = [os.path.join(CSRC, h) for h in HEADERS]
    hdr.append(os.path.join(os.path.dirname(HERE), "include", "sphq.h"))
    return [os.path.join(CSRC, s) for s in SOURCES], hdr


def up_to_date() -> bool:
    if not os.path.exists(LIB) or not os.path.exists(STUDY_LIB):
        return False
    srcs, hdrs = _inputs()
    t = min(os.path.getmtime(LIB), os.path.getmtime(STUDY_LIB))
    return all(os.path.getmtime(p) <= t for p in srcs + hdrs + [STUDY_SRC, __file__])


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    srcs, _ = _inputs()
    cc = nvcc()

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.basename(src) + ".o")
        cmd = [cc, *ARCH, *FLAGS, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        with open(obj + ".log", "w") as f:
            f.write(r.stdout + r.stderr)
        return obj

    def study():
        tmp = STUDY_LIB + f".tmp{os.getpid()}"
        cmd = [cc, *ARCH, *FLAGS, "-shared", "-o", tmp, STUDY_SRC, "-cudart", "static"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {STUDY_SRC}:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, STUDY_LIB)

    with cf.ThreadPoolExecutor(max_workers=len(srcs) + 1) as ex:
        fut = ex.submit(study)
        objs = list(ex.map(compile_one, srcs))
        fut.result()
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [cc, *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    if verbose:
        for o in objs:
            print(open(o + ".log").read())
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
