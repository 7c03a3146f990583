"""Builds the fp32 C++ oracle (flglm_oracle32.cpp) into oracle/libflglm_oracle32.so.

Test infrastructure: only the tests, the smoke check and bench.py's CPU legs load it.
Plain g++ (C++17, OpenMP, -O3; no target-specific flags, so the same source builds on
x86-64 and Arm hosts).  Rebuilds when the source is newer than the library.
"""
from __future__ import annotations

import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "flglm_oracle32.cpp")
LIB = os.path.join(HERE, "libflglm_oracle32.so")


def build(force: bool = False) -> str:
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    cxx = os.environ.get("CXX") or shutil.which("g++") or "g++"
    tmp = LIB + ".tmp"
    cmd = [cxx, "-std=c++17", "-O3", "-fopenmp", "-fPIC", "-shared", SRC, "-o", tmp]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"oracle build failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
