"""The C++ oracle (``oracle/cpp/gambit_oracle.cpp``) behind the same Python interface as the
numpy one.

``decode_attention``, ``softmax_weights``, ``probe_score``, ``running_mean_update``,
``rank_order`` and ``tournament`` have the signatures of their numpy counterparts in
``oracle.attention``, ``oracle.probe`` and ``oracle.tournament``; ``CppPool`` has the
interface of ``oracle.pool.PoolOracle`` (its per-slot arrays are numpy views of the C++
pool's own memory, so writes through them reach the pool), and ``CppBeamKV`` that of
``oracle.beams.BeamKV``.  This module only marshals arguments: every rule lives in the C++
file.  ``oracle.build_cpp`` compiles it (``__graft_entry__.build`` calls it).

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

import numpy as np

from oracle.tournament import TournamentPlan

LIB_PATH = Path(__file__).resolve().parent / "libgambit_oracle.so"
OK, ERR_INVALID, ERR_OOM, ERR_STATE = 0, 1, 2, 4

_lib = None
_P = ctypes.c_void_p
_I, _I64, _D, _F, _U32 = ctypes.c_int, ctypes.c_int64, ctypes.c_double, ctypes.c_float, ctypes.c_uint32


def load() -> ctypes.CDLL:
    """Load the C++ oracle (once); raises when it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not LIB_PATH.exists():
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m oracle.build_cpp`")
    lib = ctypes.CDLL(str(LIB_PATH))
    sig = {
        "gbo_decode_attention": ([_P, _I, _I, _P, _P, _I, _I, _D, _P], None),
        "gbo_softmax_weights": ([_P, _P, _I, _I, _D, _P], None),
        "gbo_probe_score": ([_P, _I, _I, _P, _D, _P], None),
        "gbo_running_mean_update": ([_F, _I, _F], _F),
        "gbo_tournament": ([_P, _P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _P], _I),
        "gbo_pool_new": ([_I64, _I, _I, _I], _P),
        "gbo_pool_free": ([_P], None),
        "gbo_pool_clone": ([_P], _P),
        "gbo_pool_array": ([_P, _I], _P),
        "gbo_pool_seed": ([_P, _I, _I64], _I),
        "gbo_pool_begin_step": ([_P], _I),
        "gbo_pool_status": ([_P], _I),
        "gbo_pool_set_status": ([_P, _I], None),
        "gbo_pool_set_capacity": ([_P, _I], None),
        "gbo_pool_capacity": ([_P], _I),
        "gbo_pool_num_free": ([_P], _I64),
        "gbo_pool_next_lineage": ([_P], _U32),
        "gbo_pool_prune_branch": ([_P, _I, _I, _I64, _P, _P, _P], None),
        "gbo_pool_last_plan": ([_P, _P, _P, _P, _P, _P, _P], _I),
        "gbo_pool_fork_slots": ([_P, _P], None),
        "gbo_pool_release": ([_P, _P, _I], None),
        "gbo_pool_table": ([_P, _I, _P, _I], _I),
        "gbo_pool_history": ([_P, _I, _P, _I], _I),
        "gbo_pool_cow_events": ([_P, _P, _I], _I),
        "gbo_pool_check": ([_P], ctypes.c_char_p),
        "gbo_kv_new": ([_I, _I, _I, _I], _P),
        "gbo_kv_free": ([_P], None),
        "gbo_kv_append": ([_P, _I, _I, _P, _P, _I], None),
        "gbo_kv_branch": ([_P, _I, _I], None),
        "gbo_kv_release": ([_P, _I], None),
        "gbo_kv_get": ([_P, _I, _I, _P, _P], _I),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


# ---- attention and probe ------------------------------------------------------------------------

def decode_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, scale: float) -> np.ndarray:
    """q [Hq][D], K, V [L][Hkv][D] -> o [Hq][D] fp64 (see oracle.attention.decode_attention)."""
    q, K, V = _f64(q), _f64(K), _f64(V)
    Hq, D = q.shape
    L, Hkv, D2 = K.shape
    assert D == D2 and V.shape == K.shape and L >= 1 and Hq % Hkv == 0
    out = np.empty((Hq, D), dtype=np.float64)
    load().gbo_decode_attention(_ptr(q), Hq, D, _ptr(K), _ptr(V), L, Hkv, float(scale), _ptr(out))
    return out


def softmax_weights(q: np.ndarray, K: np.ndarray, scale: float) -> np.ndarray:
    """q [D], K [L][D] -> p [L] fp64."""
    q, K = _f64(q), _f64(K)
    p = np.empty(K.shape[0], dtype=np.float64)
    load().gbo_softmax_weights(_ptr(q), _ptr(K), K.shape[0], K.shape[1], float(scale), _ptr(p))
    return p


def probe_score(h: np.ndarray, w: np.ndarray, bias: float) -> np.ndarray:
    """sigma(w.h + b) in fp64 for h [..., H]."""
    h, w = _f64(h), _f64(w)                  # held in locals: the C call reads their memory
    rows = h.reshape(-1, h.shape[-1])
    out = np.empty(rows.shape[0], dtype=np.float64)
    load().gbo_probe_score(_ptr(rows), rows.shape[0], rows.shape[1], _ptr(w), float(bias), _ptr(out))
    return out.reshape(h.shape[:-1])


def running_mean_update(mean, n: int, x) -> tuple[np.float32, int]:
    return np.float32(load().gbo_running_mean_update(float(np.float32(mean)), int(n), float(np.float32(x)))), n + 1


# ---- tournament -------------------------------------------------------------------------------------

def tournament(mean, active, eligible, capacity: int, K: int, fanout: int) -> TournamentPlan:
    if fanout < 2:
        raise ValueError("fan-out must be at least 2")
    mean = np.ascontiguousarray(mean, dtype=np.float32)
    n = len(mean)
    act = np.ascontiguousarray(np.asarray(active) != 0, dtype=np.uint8)
    elig = np.ascontiguousarray(np.asarray(eligible) != 0, dtype=np.uint8)
    kase, n_order, n_pruned = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    order = np.empty(n, np.int32)
    pruned = np.empty(n, np.int32)
    children = np.empty(2 * max(n, capacity), np.int32)
    nc = load().gbo_tournament(_ptr(mean), _ptr(act), _ptr(elig), n, int(capacity), int(K), int(fanout),
                               ctypes.byref(kase), _ptr(order), ctypes.byref(n_order), _ptr(pruned),
                               ctypes.byref(n_pruned), _ptr(children))
    return TournamentPlan(kase.value, [int(s) for s in order[:n_order.value]],
                          [int(s) for s in pruned[:n_pruned.value]],
                          [(int(children[2 * k]), int(children[2 * k + 1])) for k in range(nc)])


def rank_order(mean, active) -> list[int]:
    return tournament(mean, active, np.zeros(len(mean), np.uint8), len(mean), 0, 2).order


# ---- the pool -----------------------------------------------------------------------------------------

class CppPool:
    """The C++ pool, with the interface of oracle.pool.PoolOracle."""

    def __init__(self, num_pages: int, max_beams: int, max_pages_per_beam: int, page_size: int,
                 _handle: int | None = None):
        lib = load()
        self.num_pages = int(num_pages)
        self.max_beams = int(max_beams)
        self.max_pages = int(max_pages_per_beam)
        self.P = int(page_size)
        self._h = _handle or lib.gbo_pool_new(self.num_pages, self.max_beams, self.max_pages, self.P)

        def view(which, dtype, n):
            addr = lib.gbo_pool_array(self._h, which)
            return np.frombuffer((ctypes.c_byte * (n * np.dtype(dtype).itemsize)).from_address(addr), dtype=dtype)
        B = self.max_beams
        self.seq_len = view(0, np.int64, B)
        self.active = view(1, np.bool_, B)
        self.gen = view(2, np.int64, B)
        self.mean = view(3, np.float32, B)
        self.nsteps = view(4, np.int64, B)
        self.lineage = view(5, np.uint32, B)
        self.refcnt = view(6, np.int64, self.num_pages)

    def __del__(self):
        if getattr(self, "_h", None) and _lib is not None:
            _lib.gbo_pool_free(self._h)
            self._h = None

    def __deepcopy__(self, memo):
        return CppPool(self.num_pages, self.max_beams, self.max_pages, self.P, _handle=load().gbo_pool_clone(self._h))

    # state read back from the C++ pool
    @property
    def status(self) -> int:
        return load().gbo_pool_status(self._h)

    @status.setter
    def status(self, code: int) -> None:
        load().gbo_pool_set_status(self._h, int(code))

    @property
    def _free(self) -> list[int]:
        """Free page ids (those with no reference; check_invariants checks the C++ free set is exactly these)."""
        return [int(p) for p in np.flatnonzero(self.refcnt == 0)]

    @property
    def capacity(self) -> int:
        return load().gbo_pool_capacity(self._h)

    @capacity.setter
    def capacity(self, c: int) -> None:
        load().gbo_pool_set_capacity(self._h, int(c))

    @property
    def next_lineage(self) -> int:
        return int(load().gbo_pool_next_lineage(self._h))

    # Tables and histories are copied out of the C++ pool once per state change and cached
    # (callers index them in loops); every operation that changes them drops the copies.
    def _changed(self) -> None:
        self._tables = None
        self._history = None

    @property
    def tables(self) -> list[list[int]]:
        if getattr(self, "_tables", None) is None:
            buf = np.empty(self.max_pages + 1, np.int64)
            out = []
            for b in range(self.max_beams):
                n = load().gbo_pool_table(self._h, b, _ptr(buf), len(buf))
                out.append([int(p) for p in buf[:n]])
            self._tables = out
        return self._tables

    @property
    def history(self) -> list[list[list[int]]]:
        if getattr(self, "_history", None) is None:
            out = []
            for b in range(self.max_beams):
                n = load().gbo_pool_history(self._h, b, None, 0)
                buf = np.empty(3 * max(n, 1), np.int64)
                load().gbo_pool_history(self._h, b, _ptr(buf), n)
                out.append([[int(buf[3 * i]), int(buf[3 * i + 1]), int(buf[3 * i + 2])] for i in range(n)])
            self._history = out
        return self._history

    @property
    def cow_events(self) -> list[tuple[int, int, int, int]]:
        n = load().gbo_pool_cow_events(self._h, None, 0)
        buf = np.empty(4 * max(n, 1), np.int64)
        load().gbo_pool_cow_events(self._h, _ptr(buf), n)
        return [tuple(int(x) for x in buf[4 * i:4 * i + 4]) for i in range(n)]

    def num_free(self) -> int:
        return int(load().gbo_pool_num_free(self._h))

    def free_bits(self) -> np.ndarray:
        words = np.zeros((self.num_pages + 31) // 32, dtype=np.uint32)
        for p in np.flatnonzero(self.refcnt == 0):
            words[p // 32] |= np.uint32(1 << (p % 32))
        return words

    def check_invariants(self) -> None:
        msg = load().gbo_pool_check(self._h).decode()
        assert msg == "", msg

    # operations
    def seed(self, n_beams: int, prompt_len: int) -> None:
        from oracle.pool import PoolOOM
        assert 1 <= n_beams <= self.max_beams and prompt_len >= 1
        self._changed()
        if not load().gbo_pool_seed(self._h, int(n_beams), int(prompt_len)):
            raise PoolOOM

    def begin_step(self) -> bool:
        self._changed()
        return bool(load().gbo_pool_begin_step(self._h))

    def eligible(self, warmup: int, mask=None) -> np.ndarray:
        e = self.gen >= warmup
        if mask is not None:
            e = e & (np.asarray(mask) != 0)
        return e & self.active

    def prune_branch(self, K: int, fanout: int, warmup: int = 0, mask=None):
        if fanout < 2:
            raise ValueError("fan-out must be at least 2")
        m = None if mask is None else np.ascontiguousarray(np.asarray(mask) != 0, dtype=np.uint8)
        parent_of = np.empty(self.max_beams, np.int32)
        pruned = np.empty(self.max_beams, np.uint8)
        self._changed()
        load().gbo_pool_prune_branch(self._h, int(K), int(fanout), int(warmup), None if m is None else _ptr(m),
                                     _ptr(parent_of), _ptr(pruned))
        n_order, n_pruned, n_children = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
        order = np.empty(self.max_beams, np.int32)
        pr = np.empty(self.max_beams, np.int32)
        ch = np.empty(2 * self.max_beams, np.int32)
        kase = load().gbo_pool_last_plan(self._h, _ptr(order), ctypes.byref(n_order), _ptr(pr), ctypes.byref(n_pruned),
                                         _ptr(ch), ctypes.byref(n_children))
        plan = TournamentPlan(kase, [int(s) for s in order[:n_order.value]], [int(s) for s in pr[:n_pruned.value]],
                              [(int(ch[2 * k]), int(ch[2 * k + 1])) for k in range(n_children.value)])
        return plan, parent_of.astype(np.int64), pruned

    def fork_slots(self, parent_of) -> None:
        p = np.ascontiguousarray(parent_of, dtype=np.int32)
        self._changed()
        load().gbo_pool_fork_slots(self._h, _ptr(p))

    def release(self, slots) -> None:
        s = np.ascontiguousarray(np.asarray(slots, dtype=np.int64), dtype=np.int32)
        self._changed()
        load().gbo_pool_release(self._h, _ptr(s) if len(s) else None, len(s))


class CppBeamKV:
    """Every beam's full K/V kept by the C++ oracle, copied on branch (interface of oracle.beams.BeamKV)."""

    def __init__(self, num_layers: int, max_beams: int, num_kv_heads: int, head_dim: int):
        self.layers, self.Hkv, self.D = num_layers, num_kv_heads, head_dim
        self._h = load().gbo_kv_new(num_layers, max_beams, num_kv_heads, head_dim)

    def __del__(self):
        if getattr(self, "_h", None) and _lib is not None:
            _lib.gbo_kv_free(self._h)
            self._h = None

    def append_rows(self, slot: int, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        k = np.ascontiguousarray(k, dtype=np.float32).reshape(-1, self.Hkv, self.D)
        v = np.ascontiguousarray(v, dtype=np.float32).reshape(-1, self.Hkv, self.D)
        load().gbo_kv_append(self._h, int(slot), int(layer), _ptr(k), _ptr(v), k.shape[0])

    def seed(self, n_beams: int, k_prompt: list, v_prompt: list) -> None:
        for b in range(n_beams):
            for layer in range(self.layers):
                self.append_rows(b, layer, k_prompt[layer], v_prompt[layer])

    def append(self, slot: int, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        self.append_rows(slot, layer, k[None], v[None])

    def branch(self, child: int, parent: int) -> None:
        load().gbo_kv_branch(self._h, int(child), int(parent))

    def release(self, slot: int) -> None:
        load().gbo_kv_release(self._h, int(slot))

    def get(self, slot: int, layer: int) -> tuple[np.ndarray, np.ndarray]:
        n = load().gbo_kv_get(self._h, int(slot), int(layer), None, None)
        K = np.empty((n, self.Hkv, self.D), np.float64)
        V = np.empty((n, self.Hkv, self.D), np.float64)
        load().gbo_kv_get(self._h, int(slot), int(layer), _ptr(K), _ptr(V))
        return K, V
