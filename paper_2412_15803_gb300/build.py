"""Builds libwq4.so (the CUDA library behind include/wq4.h) in-tree.

    python -m paper_2412_15803_gb300.build [--force] [--verbose]

nvcc compiles each translation unit for sm_103a only, in parallel, and links
them into paper_2412_15803_gb300/_build/libwq4.so against the shared CUDA
runtime.  ptxas resource usage (-Xptxas -v) is written next to the objects.
"""
from __future__ import annotations

import argparse
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD, "libwq4.so")

SOURCES = ["wq4_gemv.cu", "wq4_chain.cu", "wq4_synth.cu", "wq4_tc.cu", "wq4_attn.cu", "wq4_gemm.cu"]
HEADERS = ["wq4_device.cuh", "wq4_host.h", "wq4_items.cuh", "wq4_tc.cuh", "wq4_tc_host.h"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    return cand


def cuda_lib_dir() -> str:
    root = os.path.dirname(os.path.dirname(os.path.realpath(nvcc())))
    for d in ("lib64", os.path.join("targets", "sbsa-linux", "lib"), os.path.join("targets", "x86_64-linux", "lib")):
        p = os.path.join(root, d)
        if os.path.isdir(p):
            return p
    return os.path.join(root, "lib64")


def _inputs():
    files = [os.path.join(CSRC, s) for s in SOURCES + HEADERS]
    files += [os.path.join(INCLUDE, h) for h in ("wq4.h", "wq4_synth.h", "wq4_attn.h")]
    files.append(os.path.abspath(__file__))
    return files


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    common = [nvcc(), *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
              "-I", INCLUDE, "-I", CSRC, "-Xptxas", "-v"]
    procs = []
    for src in SOURCES:
        obj = os.path.join(BUILD, src.replace(".cu", ".o"))
        log = open(os.path.join(BUILD, src.replace(".cu", ".ptxas.txt")), "w")
        cmd = common + ["-c", os.path.join(CSRC, src), "-o", obj]
        procs.append((src, obj, subprocess.Popen(cmd, stdout=log, stderr=subprocess.STDOUT), log))
    objs = []
    failed = []
    for src, obj, p, log in procs:
        rc = p.wait()
        log.close()
        if rc != 0:
            failed.append(src)
        objs.append(obj)
        if verbose or rc != 0:
            sys.stderr.write(open(log.name).read())
    if failed:
        raise RuntimeError("nvcc failed for " + ", ".join(failed))
    tmp = LIB + f".tmp{os.getpid()}"
    libdir = cuda_lib_dir()
    subprocess.check_call([nvcc(), *ARCH, "-shared", "-cudart", "shared", "-o", tmp, *objs,
                           "-L", libdir, f"-Xlinker=-rpath={libdir}"])
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    ap = argparse.ArgumentParser()
    ap.add_argument("--force", action="store_true")
    ap.add_argument("--verbose", action="store_true")
    a = ap.parse_args()
    print(build(force=a.force, verbose=a.verbose))
