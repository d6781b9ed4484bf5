"""ctypes binding of ``workload/libgbgen.so``: the device-side seeded generator.

Produces exactly the values of ``workload.gen`` (checked bit for bit by
``tests/test_gpu_gen.py``) directly in device memory, for inputs too large to
generate on the host.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

from workload import gen

LIB_PATH = Path(__file__).resolve().with_name("libgbgen.so")
_lib = None


def load() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not LIB_PATH.exists():
            raise RuntimeError(f"{LIB_PATH} is missing: run the build first")
        _lib = ctypes.CDLL(str(LIB_PATH))
        _lib.gbgen_normal.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                      ctypes.c_int, ctypes.POINTER(ctypes.c_longlong), ctypes.c_float,
                                      ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p]
        _lib.gbgen_normal.restype = ctypes.c_int
    return _lib


def _signed(x: int) -> int:
    x &= (1 << 64) - 1
    return x - (1 << 64) if x >= (1 << 63) else x


def normal(out, dtype: str, n0: int, n1: int, n2: int, fields: list, scale: float = 1.0, row_scale=None,
           row_scale_div: int = 1, stream=None) -> None:
    """out[(i0*n1 + i1)*n2 + j] = normal(key(fields(i0, i1)), j) * scale [* row_scale[j // div]].

    Each field is an int (constant) or a tuple (base, c0, c1): base + c0*i0 + c1*i1.
    """
    flat = []
    for f in fields:
        if isinstance(f, tuple):
            b, c0, c1 = f
        else:
            b, c0, c1 = f, 0, 0
        flat += [_signed(int(b)), _signed(int(c0)), _signed(int(c1))]
    arr = (ctypes.c_longlong * len(flat))(*flat)
    rs = row_scale.data_ptr() if row_scale is not None else None
    st = stream.cuda_stream if stream is not None and not isinstance(stream, int) else stream
    if st is None:
        import torch
        st = torch.cuda.current_stream().cuda_stream
    code = load().gbgen_normal(out.data_ptr(), 1 if dtype == "bf16" else 0, n0, n1, n2, len(fields), arr,
                               float(scale), rs, row_scale_div, st)
    if code != 0:
        raise RuntimeError(f"gbgen_normal failed with CUDA error {code}")


__all__ = ["normal", "load", "gen"]
