"""In-tree build of libkvc.so (sm_103a) with nvcc; translation units compile in parallel."""
from __future__ import annotations

import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "_build")
SO = os.path.join(OUT, "libkvc.so")
INCLUDE = os.path.join(ROOT, "include")
GENCODE = "arch=compute_103a,code=sm_103a"
SOURCES = ["kvc.cpp", "book.cpp", "kernels.cu", "prefill.cu"]
HEADERS = [os.path.join(CSRC, h) for h in ("book.hpp", "kernels.hpp", "device_common.cuh")] + [os.path.join(INCLUDE, "kvc.h")]


def _flags(verbose_ptx: bool = False):
    f = ["nvcc", "-gencode", GENCODE, "-lineinfo", "-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE]
    if verbose_ptx:
        f += ["-Xptxas", "-v"]
    return f


def _stale() -> bool:
    if not os.path.exists(SO):
        return True
    t = os.path.getmtime(SO)
    deps = [os.path.join(CSRC, s) for s in SOURCES] + HEADERS
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose_ptx: bool = False) -> str:
    if not (force or verbose_ptx or _stale()):
        return SO
    os.makedirs(OUT, exist_ok=True)

    def compile_one(src):
        obj = os.path.join(OUT, src + f".{os.getpid()}.o")
        cmd = _flags(verbose_ptx) + ["-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with ThreadPoolExecutor(len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose_ptx:
        for _, log in results:
            print(log)
    objs = [o for o, _ in results]
    tmp = SO + f".{os.getpid()}.tmp"
    r = subprocess.run(["nvcc", "-gencode", GENCODE, "-shared", "-o", tmp] + objs + ["-lcudart"], capture_output=True,
                       text=True)
    for o in objs:
        os.remove(o)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, SO)
    return SO


if __name__ == "__main__":
    import sys

    print(build(force=True, verbose_ptx="-v" in sys.argv))
