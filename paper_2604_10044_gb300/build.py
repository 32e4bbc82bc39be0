"""Build of liblg.so: every .cu of csrc/ compiled for sm_103a in parallel, then linked.

The library links the CUDA runtime statically and exports only the lg_* C ABI declared in
include/lg.h.
"""
import os
import subprocess

_HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(_HERE)
CSRC = os.path.join(_HERE, "csrc")
BUILD = os.path.join(_HERE, "_build")
LIB = os.path.join(_HERE, "liblg.so")
SOURCES = ["lg_attend.cu", "lg_attend_mma.cu", "lg_guard.cu", "lg_token.cu", "lg_api.cu",
           "lg_noalloc.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-fvisibility=hidden",
         "-I" + os.path.join(ROOT, "include"), "-I" + CSRC]


def _obj(src):
    return os.path.join(BUILD, os.path.splitext(src)[0] + ".o")


def build_async(extra=()):
    """start one nvcc per translation unit; returns the Popen handles"""
    os.makedirs(BUILD, exist_ok=True)
    procs = []
    for src in SOURCES:
        cmd = ["nvcc"] + ARCH + FLAGS + list(extra) + ["-c", os.path.join(CSRC, src), "-o",
                                                       _obj(src)]
        procs.append(subprocess.Popen(cmd))
    return procs


def link():
    cmd = ["nvcc"] + ARCH + ["-shared", "-o", LIB] + [_obj(s) for s in SOURCES]
    return subprocess.call(cmd)


def build():
    procs = build_async()
    if any(p.wait() != 0 for p in procs):
        raise RuntimeError("nvcc failed")
    if link() != 0:
        raise RuntimeError("link failed")
