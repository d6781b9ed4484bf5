"""Compile the C++ oracle (``oracle/cpp/gambit_oracle.cpp``) into ``oracle/libgambit_oracle.so``
with the host compiler: plain C++17, no CUDA, no architecture-specific flags, floating-point
contraction off (the running mean's operations are rounded one by one).

Building the oracle is part of building the test infrastructure; nothing in the product
loads it.
"""
from __future__ import annotations

import os
import platform
import subprocess
import sys
from pathlib import Path

HERE = Path(__file__).resolve().parent
SRC = HERE / "cpp" / "gambit_oracle.cpp"
LIB = HERE / "libgambit_oracle.so"
STAMP = HERE / "cpp" / ".built_for"


def build(force: bool = False) -> Path:
    arch = platform.machine()
    fresh = LIB.exists() and STAMP.exists() and STAMP.read_text() == arch and \
        LIB.stat().st_mtime >= SRC.stat().st_mtime
    if fresh and not force:
        return LIB
    cxx = os.environ.get("CXX", "g++")
    cmd = [cxx, "-std=c++17", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-o", str(LIB), str(SRC)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        sys.stderr.write(r.stdout + r.stderr)
        raise RuntimeError(f"oracle build failed: {' '.join(cmd)}")
    STAMP.write_text(arch)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
