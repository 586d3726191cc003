"""Build libcmsd.so (and the decode-simulation workload library) for sm_103a.

Plain nvcc, one object per translation unit compiled in parallel, linked in
place next to this file (no install step).  Object files go to <repo>/_build.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OBJDIR = os.path.join(ROOT, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I" + INCLUDE, "-I" + CSRC]

LIBS = {
    "libcmsd.so": ["cmsd_stream_bf16.cu", "cmsd_stream_f32.cu", "cmsd_api.cu", "cmsd_static.cu", "cmsd_lmhead.cu"],
    "libcmsd_workload.so": ["cmsd_workload.cu"],
}


def nvcc_path():
    p = shutil.which("nvcc")
    if p:
        return p
    cand = "/usr/local/cuda/bin/nvcc"
    if os.path.exists(cand):
        return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libcmsd.so")


def _run(cmd, verbose):
    if verbose:
        print(" ".join(cmd), flush=True)
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("command failed: %s\n%s%s" % (" ".join(cmd), r.stdout, r.stderr))
    return r.stdout + r.stderr


def build(verbose=False, ptxas_info=False):
    """Compile every CUDA library of the package; returns the built paths."""
    nvcc = nvcc_path()
    os.makedirs(OBJDIR, exist_ok=True)
    jobs = []
    for lib, srcs in LIBS.items():
        for s in srcs:
            src = os.path.join(CSRC, s)
            if not os.path.exists(src):
                continue
            obj = os.path.join(OBJDIR, s.replace(".cu", ".o"))
            cmd = [nvcc] + ARCH + NVCC_FLAGS + (["-Xptxas", "-v"] if ptxas_info else []) + ["-c", src, "-o", obj]
            jobs.append(cmd)
    with ThreadPoolExecutor(max_workers=min(8, max(1, len(jobs)))) as ex:
        logs = list(ex.map(lambda c: _run(c, verbose), jobs))
    if ptxas_info:
        for log in logs:
            sys.stdout.write(log)
    built = []
    for lib, srcs in LIBS.items():
        objs = [os.path.join(OBJDIR, s.replace(".cu", ".o")) for s in srcs
                if os.path.exists(os.path.join(CSRC, s))]
        if not objs:
            continue
        out = os.path.join(PKG, lib)
        tmp = out + ".tmp"
        _run([nvcc] + ARCH + ["-shared", "-o", tmp] + objs, verbose)
        os.replace(tmp, out)
        built.append(out)
    return built


if __name__ == "__main__":
    for p in build(verbose="-v" in sys.argv, ptxas_info="--ptxas" in sys.argv):
        print(p)
