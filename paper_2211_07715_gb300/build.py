"""Compile libbsgemm.so in-tree with nvcc for sm_103a (GB300).

Six translation units (layer kernels, pruning kernel, attention kernel, sparse tensor-core kernel, int8 peak probes, host ABI) compile in parallel, then link
into one shared library with the CUDA runtime linked statically, so the
library needs nothing but the NVIDIA driver at run time.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import tempfile

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(PKG, "libbsgemm.so")
SOURCES = ["bsgemm_kernel.cu", "bsgemm_prune.cu", "bsgemm_attention.cu", "bsgemm_sparse24.cu", "bsgemm_peaks.cu",
           "bsgemm_api.cpp"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found; the CUDA 13 toolkit is required to build libbsgemm.so")


def _inputs():
    files = [os.path.join(CSRC, s) for s in SOURCES] + [os.path.join(CSRC, h) for h in ("bsgemm_device.cuh", "bsgemm_tcgen05.cuh")]
    files += [os.path.join(CSRC, "bsgemm_internal.h"), os.path.join(INCLUDE, "bsgemm.h")]
    return files


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and up_to_date():
        return LIB
    cc = nvcc()
    common = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC]
    if verbose:
        common += ["-Xptxas", "-v"]
    with tempfile.TemporaryDirectory(prefix="bsgemm_build_") as tmp:
        objs, procs = [], []
        for src in SOURCES:
            obj = os.path.join(tmp, src + ".o")
            objs.append(obj)
            procs.append((src, subprocess.Popen([cc, *common, "-c", os.path.join(CSRC, src), "-o", obj],
                                                stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
        for src, p in procs:
            out, _ = p.communicate()
            if verbose and out:
                print(out)
            if p.returncode != 0:
                raise RuntimeError(f"nvcc failed on {src}:\n{out}")
        tmp_lib = os.path.join(tmp, "libbsgemm.so")
        subprocess.check_call([cc, *ARCH, "-shared", "-Xcompiler", "-fPIC", *objs, "-o", tmp_lib])
        shutil.copyfile(tmp_lib, LIB + ".tmp")
        os.replace(LIB + ".tmp", LIB)
    return LIB


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
