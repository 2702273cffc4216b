"""Compiles the CPU oracle (oracle.c) into oracle/liboracle.so with gcc (test infrastructure)."""
from __future__ import annotations

import os
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
SRCS = [HERE / "oracle.c", HERE / "oracle.h"]
LIB = HERE / "liboracle.so"


def build(force: bool = False) -> Path:
    newest = max(p.stat().st_mtime for p in SRCS)
    if not force and LIB.exists() and LIB.stat().st_mtime >= newest:
        return LIB
    tmp = LIB.with_suffix(f".so.tmp{os.getpid()}")
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           str(HERE / "oracle.c"), "-o", str(tmp), "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
