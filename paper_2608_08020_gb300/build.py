"""Build the CUDA libraries in-tree with nvcc for sm_103a.

* ``paper_2608_08020_gb300/libgambit.so`` - the beam-decode library (C ABI in
  ``include/gambit.h``), compiled from ``paper_2608_08020_gb300/csrc/*.cu``.
* ``workload/libgbgen.so`` - the device-side seeded input generator.

Translation units compile in parallel; objects go to ``_build/`` (git-ignored).
"""
from __future__ import annotations

import os
import platform
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor
from pathlib import Path

ROOT = Path(__file__).resolve().parent.parent
PKG = ROOT / "paper_2608_08020_gb300"
CSRC = PKG / "csrc"
INCLUDE = ROOT / "include"
BUILD = ROOT / "_build" / platform.machine()   # objects of another host architecture are never reused
LIB = PKG / "libgambit.so"
GEN_SRC = ROOT / "workload" / "gen.cu"
GEN_LIB = ROOT / "workload" / "libgbgen.so"

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
                     "-I", str(INCLUDE)]


LINK_FLAGS = ["-shared", "-cudart", "shared", "-Xlinker", "-rpath", "-Xlinker", "/usr/local/cuda/lib64"]


def _nvcc() -> str:
    cand = os.environ.get("NVCC") or "/usr/local/cuda/bin/nvcc"
    return cand if Path(cand).exists() else "nvcc"


def _run(cmd: list[str], verbose: bool) -> None:
    if verbose:
        print(" ".join(cmd), flush=True)
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        sys.stderr.write(r.stdout + r.stderr)
        raise RuntimeError(f"command failed ({r.returncode}): {' '.join(cmd)}")
    if verbose and (r.stdout or r.stderr):
        print(r.stdout + r.stderr, flush=True)


def _stale(target: Path, deps: list[Path]) -> bool:
    if not target.exists():
        return True
    t = target.stat().st_mtime
    return any(d.stat().st_mtime > t for d in deps)


def build(verbose: bool = False, force: bool = False, extra_flags: list[str] | None = None) -> None:
    nvcc = _nvcc()
    BUILD.mkdir(parents=True, exist_ok=True)
    flags = NVCC_FLAGS + list(extra_flags or [])
    headers = list(CSRC.glob("*.cuh")) + [INCLUDE / "gambit.h"]
    sources = sorted(CSRC.glob("*.cu"))
    jobs = []
    objs = []
    for src in sources:
        obj = BUILD / (src.stem + ".o")
        objs.append(obj)
        if force or _stale(obj, [src] + headers):
            jobs.append([nvcc] + flags + ["-c", str(src), "-o", str(obj)])
    gen_obj = BUILD / "gen.o"
    if force or _stale(gen_obj, [GEN_SRC]):
        jobs.append([nvcc] + flags + ["-c", str(GEN_SRC), "-o", str(gen_obj)])
    with ThreadPoolExecutor(max_workers=max(1, min(len(jobs), os.cpu_count() or 4))) as ex:
        list(ex.map(lambda c: _run(c, verbose), jobs))
    stamp = BUILD / "link.stamp"           # the .so must have been linked on this architecture
    if not stamp.exists():
        force = True
    if force or _stale(LIB, objs):
        _run([nvcc] + ARCH + LINK_FLAGS + ["-o", str(LIB)] + [str(o) for o in objs], verbose)
    if force or _stale(GEN_LIB, [gen_obj]):
        _run([nvcc] + ARCH + LINK_FLAGS + ["-o", str(GEN_LIB), str(gen_obj)], verbose)
    stamp.write_text(platform.machine())


if __name__ == "__main__":
    build(verbose=True, force="--force" in sys.argv)
