"""Build the CPU oracle (test infrastructure only) into oracle/_build/liboracle.so.

Plain g++: C++17, -O2, no fused multiply-add (-ffp-contract=off) and no fast-math, so the
fp64 arithmetic is IEEE and follows the written order of operations on x86-64 and aarch64
alike.  OpenMP is used for the loss rows when the compiler supports it.
"""
from __future__ import annotations

import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SOURCES = ["advantage.cpp", "mdap.cpp", "compact.cpp", "loss.cpp", "lmhead.cpp", "ars.cpp"]
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "liboracle.so")


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    deps = SOURCES + ["oracle.h"]
    return any(os.path.getmtime(os.path.join(HERE, s)) > t for s in deps)


def build_oracle(force: bool = False) -> str:
    """Compile the oracle if it is missing or older than its sources; return the .so path."""
    if not force and not _stale():
        return LIB
    os.makedirs(OUT_DIR, exist_ok=True)
    srcs = [os.path.join(HERE, s) for s in SOURCES]
    tmp = LIB + ".tmp.%d" % os.getpid()
    base = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
            "-shared", "-o", tmp] + srcs
    for extra in (["-fopenmp"], []):
        r = subprocess.run(base + extra, capture_output=True, text=True)
        if r.returncode == 0:
            os.replace(tmp, LIB)
            return LIB
    sys.stderr.write(r.stderr)
    raise RuntimeError("oracle build failed")


if __name__ == "__main__":
    print(build_oracle(force="--force" in sys.argv))
