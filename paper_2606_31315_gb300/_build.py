"""Builds libblockpilot.so in-tree with nvcc for sm_103a (translation units compiled in parallel).

Beside it, libblockpilot_shortwait.so: the same sources built with BP_TEST_SHORT_WAITS, where every
bounded wait for work to arrive is a single non-blocking test.  It exists only for the test of the
kernels' wind-down path (an expired wait reports BP_ERR_TIMEOUT, drains the kernel's own copies and
tensor-core operations, releases tensor memory and returns); nothing else loads it.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libblockpilot.so")
TEST_LIB = os.path.join(PKG, "libblockpilot_shortwait.so")  # test-only build (see above)
SOURCES = ("api.cu", "attention.cu", "accept.cu", "accept_batch.cu", "policy.cu", "verify_epilogue.cu", "verify_stream.cu", "tau.cu", "commit.cu")
HEADERS = ("common.cuh", "ptx_sm103.cuh", "softmax_math.cuh")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libblockpilot")


def _inputs_mtime() -> float:
    files = [os.path.join(CSRC, f) for f in SOURCES + HEADERS]
    files.append(os.path.join(os.path.dirname(PKG), "include", "blockpilot.h"))
    files.append(os.path.abspath(__file__))
    return max(os.path.getmtime(f) for f in files)


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile and link both libraries; returns the path of the product library."""
    stale = force or not all(os.path.exists(x) and os.path.getmtime(x) >= _inputs_mtime() for x in (LIB, TEST_LIB))
    if not stale:
        return LIB
    os.makedirs(os.path.join(BUILD, "shortwait"), exist_ok=True)
    nvcc = _nvcc()

    def compile_one(job) -> str:
        src, test = job
        obj = os.path.join(BUILD, "shortwait" if test else "", src.replace(".cu", ".o"))
        cmd = [nvcc, *ARCH, *FLAGS, *(["-DBP_TEST_SHORT_WAITS"] if test else []), "-c", os.path.join(CSRC, src), "-o",
               obj]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}{' (short waits)' if test else ''}:\n{res.stdout}\n{res.stderr}")
        if verbose:
            print(res.stdout + res.stderr)
        return obj

    jobs = [(src, test) for test in (False, True) for src in SOURCES]
    with cf.ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        objs = list(ex.map(compile_one, jobs))
    for lib, part in ((LIB, objs[:len(SOURCES)]), (TEST_LIB, objs[len(SOURCES):])):
        tmp = lib + f".tmp{os.getpid()}"
        res = subprocess.run([nvcc, *ARCH, "-shared", *part, "-o", tmp], capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"link failed:\n{res.stdout}\n{res.stderr}")
        os.replace(tmp, lib)
    return LIB


if __name__ == "__main__":  # pragma: no cover
    import sys

    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
