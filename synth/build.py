"""Build step for the synthetic input generator (host C and device CUDA builds)."""
from __future__ import annotations

import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
OUT = os.path.join(HERE, "_build")
HOST_SO = os.path.join(OUT, "libsynth_host.so")
CUDA_SO = os.path.join(OUT, "libsynth_cuda.so")
GENCODE = "arch=compute_103a,code=sm_103a"


def _stale(target: str, sources) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(os.path.join(HERE, s)) > t for s in sources)


def build_host(force: bool = False) -> str:
    srcs = ["synth_host.c", "synth_gen.h"]
    if force or _stale(HOST_SO, srcs):
        os.makedirs(OUT, exist_ok=True)
        tmp = HOST_SO + f".{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                        os.path.join(HERE, "synth_host.c"), "-o", tmp], check=True)
        os.replace(tmp, HOST_SO)
    return HOST_SO


def build_cuda(force: bool = False) -> str:
    srcs = ["synth_cuda.cu", "synth_gen.h"]
    if force or _stale(CUDA_SO, srcs):
        os.makedirs(OUT, exist_ok=True)
        tmp = CUDA_SO + f".{os.getpid()}.tmp"
        subprocess.run(["nvcc", "-gencode", GENCODE, "-lineinfo", "-O3", "-Xcompiler", "-fPIC", "-shared",
                        os.path.join(HERE, "synth_cuda.cu"), "-o", tmp], check=True)
        os.replace(tmp, CUDA_SO)
    return CUDA_SO


def build(force: bool = False):
    return build_host(force), build_cuda(force)
