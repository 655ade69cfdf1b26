"""Build step for the CPU oracle (plain C + OpenMP).  Test infrastructure only."""
from __future__ import annotations

import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
OUT = os.path.join(HERE, "_build")
SO = os.path.join(OUT, "liboracle.so")
SRC = os.path.join(HERE, "kvc_oracle.c")


def build(force: bool = False) -> str:
    if force or not os.path.exists(SO) or os.path.getmtime(SRC) > os.path.getmtime(SO):
        os.makedirs(OUT, exist_ok=True)
        tmp = SO + f".{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared", SRC, "-o",
                        tmp, "-lm"], check=True)
        os.replace(tmp, SO)
    return SO
