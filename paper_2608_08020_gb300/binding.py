"""ctypes binding of ``libgambit.so`` (the C ABI declared in ``include/gambit.h``).

Argument marshalling only: every step of the hot path runs in the library's
CUDA kernels.  Device arguments may be torch tensors (their ``data_ptr()`` is
passed) or raw integer device addresses; streams may be ``torch.cuda.Stream``
objects, raw ``cudaStream_t`` integers or ``None`` (the current torch stream
when torch is initialised on CUDA, else the legacy default stream).

If the shared library has not been built the import of this module succeeds
but the first call raises ``RuntimeError``: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

LIB_PATH = Path(__file__).resolve().with_name("libgambit.so")

GB_OK, GB_ERR_INVALID, GB_ERR_OOM, GB_ERR_CUDA, GB_ERR_STATE, GB_ERR_TIMEOUT, GB_ERR_UNSUPPORTED = range(7)
GB_ERR_TOO_LARGE = 7
STATUS_NAMES = {0: "GB_OK", 1: "GB_ERR_INVALID", 2: "GB_ERR_OOM", 3: "GB_ERR_CUDA", 4: "GB_ERR_STATE",
                5: "GB_ERR_TIMEOUT", 6: "GB_ERR_UNSUPPORTED", 7: "GB_ERR_TOO_LARGE"}
GB_F32, GB_BF16 = 0, 1
STATS_WORDS = 10  # words per record of gb_pool_read_step_stats
GB_PATH_AUTO, GB_PATH_PER_BEAM, GB_PATH_GROUPED = 0, 1, 2

# Every symbol the header declares, in header order.
EXPORTS = ["gb_pool_workspace_bytes", "gb_pool_init", "gb_pool_destroy", "gb_pool_seed", "gb_decode_attention",
           "gb_append_kv", "gb_score_probe", "gb_push_scores", "gb_prune_branch", "gb_release", "gb_pool_status",
           "gb_pool_clear_status", "gb_pool_wait_selftest", "gb_pool_read_state", "gb_pool_set_profile_events", "gb_pool_launch_count",
           "gb_paged_decode_noalloc", "gb_paged_decode_noalloc_status", "gb_pool_read_step_stats", "gb_pool_set_capacity", "gb_pool_last_ranked", "gb_score_mlp", "gb_fork_slots", "gb_scorer_sizes", "gb_scorer_seed",
           "gb_scorer_step", "gb_last_error"]
GB_PROF_DECODE, GB_PROF_PROBE, GB_PROF_PRUNE, GB_PROF_GROUPED = 0, 1, 2, 3
GB_PROF_PLAN, GB_PROF_APPEND, GB_PROF_COMBINE, GB_PROF_ATTENTION = 4, 5, 6, 7


class GbPoolConfig(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int), ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("page_size", ctypes.c_int), ("kv_dtype", ctypes.c_int),
                ("num_pages", ctypes.c_int64), ("max_beams", ctypes.c_int), ("max_pages_per_beam", ctypes.c_int),
                ("group_min_beams", ctypes.c_int)]


class GbPoolState(ctypes.Structure):
    _fields_ = [("tables", ctypes.c_void_p), ("seq_len", ctypes.c_void_p), ("active", ctypes.c_void_p),
                ("gen", ctypes.c_void_p), ("nsteps", ctypes.c_void_p), ("mean", ctypes.c_void_p),
                ("lineage", ctypes.c_void_p), ("refcnt", ctypes.c_void_p), ("free_bits", ctypes.c_void_p),
                ("seg_cover", ctypes.c_void_p), ("seg_nseg", ctypes.c_void_p)]


class GbPagedDecodeArgs(ctypes.Structure):
    _fields_ = [("kv", ctypes.c_void_p), ("tables", ctypes.c_void_p), ("seq_len", ctypes.c_void_p),
                ("q", ctypes.c_void_p), ("out", ctypes.c_void_p), ("num_beams", ctypes.c_int),
                ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("page_size", ctypes.c_int), ("kv_dtype", ctypes.c_int), ("max_pages_per_beam", ctypes.c_int),
                ("num_pages", ctypes.c_int64), ("scale", ctypes.c_float)]


class GambitError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {what}")
        self.code = code


_lib = None


def load(path: Path | None = None) -> ctypes.CDLL:
    """Load the library (once).  Raises RuntimeError when it has not been built."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = Path(path) if path else LIB_PATH
    if not p.exists():
        raise RuntimeError(f"{p} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(str(p))
    V, I, F, P = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_void_p
    sig = {
        "gb_pool_workspace_bytes": [P, P, P],
        "gb_pool_init": [P, V, V, V, P],
        "gb_pool_destroy": [V],
        "gb_pool_seed": [V, I, I, V, V, V],
        "gb_decode_attention": [V, I, V, V, V, F, V, I, V],
        "gb_append_kv": [V, I, I, V, V, V],
        "gb_score_probe": [V, V, I, I, V, F, V, V, V],
        "gb_push_scores": [V, V, V, V],
        "gb_prune_branch": [V, I, I, I, V, V, V, V, V],
        "gb_release": [V, V, I, V],
        "gb_pool_status": [V, P, V],
        "gb_pool_clear_status": [V, V],
        "gb_pool_wait_selftest": [V, V],
        "gb_pool_read_state": [V, P, V],
        "gb_pool_set_profile_events": [V, I, V, V],
        "gb_pool_launch_count": [V, P],
        "gb_paged_decode_noalloc": [P, V],
        "gb_paged_decode_noalloc_status": [P, V],
        "gb_pool_read_step_stats": [V, P, I, P, V],
        "gb_pool_set_capacity": [V, I],
        "gb_pool_last_ranked": [V, V, V],
        "gb_score_mlp": [V, V, I, V, V, V, F, I, V, V, V],
        "gb_fork_slots": [V, V, V],
        "gb_scorer_sizes": [V, P, P, P, P, I, P],
        "gb_scorer_seed": [V, P, V, V, V, I, V],
        "gb_scorer_step": [V, P, V, V, V, V, V],
        "gb_last_error": [V],
    }
    for name, args in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = ctypes.c_char_p if name == "gb_last_error" else ctypes.c_int
    if path is None:
        _lib = lib
    return lib


def ptr(x) -> int | None:
    """Device address of a tensor / int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def stream_handle(s) -> int | None:
    if s is None:
        try:
            import torch
            if torch.cuda.is_available() and torch.cuda.is_initialized():
                return torch.cuda.current_stream().cuda_stream
        except Exception:
            pass
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(pool_handle, code: int, what: str) -> None:
    if code != GB_OK:
        detail = load().gb_last_error(pool_handle) if pool_handle else b""
        raise GambitError(code, f"{what}: {(detail or b'').decode()}")


# ---------------------------------------------------------------------------
# Functions with the C names (raise GambitError on a non-OK status).
# ---------------------------------------------------------------------------

def gb_pool_workspace_bytes(cfg: GbPoolConfig) -> tuple[int, int]:
    kv, meta = ctypes.c_size_t(), ctypes.c_size_t()
    _check(None, load().gb_pool_workspace_bytes(ctypes.byref(cfg), ctypes.byref(kv), ctypes.byref(meta)),
           "gb_pool_workspace_bytes")
    return kv.value, meta.value


def gb_pool_init(cfg: GbPoolConfig, kv_dev, meta_dev, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(None, load().gb_pool_init(ctypes.byref(cfg), ptr(kv_dev), ptr(meta_dev), stream_handle(stream),
                                     ctypes.byref(h)), "gb_pool_init")
    return h.value


def gb_pool_destroy(pool: int) -> None:
    load().gb_pool_destroy(pool)


def gb_pool_seed(pool: int, n_beams: int, prompt_len: int, k_prompt, v_prompt, stream=None) -> None:
    _check(pool, load().gb_pool_seed(pool, n_beams, prompt_len, ptr(k_prompt), ptr(v_prompt),
                                     stream_handle(stream)), "gb_pool_seed")


def gb_decode_attention(pool: int, layer: int, q, k_new, v_new, scale: float, out, flags: int = GB_PATH_AUTO,
                        stream=None) -> None:
    _check(pool, load().gb_decode_attention(pool, layer, ptr(q), ptr(k_new), ptr(v_new), float(scale), ptr(out),
                                            flags, stream_handle(stream)), "gb_decode_attention")


def gb_append_kv(pool: int, layer: int, n_tokens: int, k, v, stream=None) -> None:
    _check(pool, load().gb_append_kv(pool, layer, n_tokens, ptr(k), ptr(v), stream_handle(stream)), "gb_append_kv")


def gb_score_probe(pool: int, hidden, hidden_dtype: int, hidden_dim: int, w, bias: float, mask=None,
                   score_out=None, stream=None) -> None:
    _check(pool, load().gb_score_probe(pool, ptr(hidden), hidden_dtype, hidden_dim, ptr(w), float(bias), ptr(mask),
                                       ptr(score_out), stream_handle(stream)), "gb_score_probe")


def gb_score_mlp(pool: int, hidden, hidden_dim: int, w1, b1, w2, b2: float, d_h: int, mask=None, score_out=None,
                 stream=None) -> None:
    _check(pool, load().gb_score_mlp(pool, ptr(hidden), hidden_dim, ptr(w1), ptr(b1), ptr(w2), float(b2), d_h,
                                     ptr(mask), ptr(score_out), stream_handle(stream)), "gb_score_mlp")


def gb_push_scores(pool: int, scores, mask=None, stream=None) -> None:
    _check(pool, load().gb_push_scores(pool, ptr(scores), ptr(mask), stream_handle(stream)), "gb_push_scores")


def gb_prune_branch(pool: int, K: int, fanout: int, warmup: int = 0, eligible=None, parent_out=None,
                    pruned_out=None, lineage_out=None, stream=None) -> None:
    _check(pool, load().gb_prune_branch(pool, K, fanout, warmup, ptr(eligible), ptr(parent_out), ptr(pruned_out),
                                        ptr(lineage_out), stream_handle(stream)), "gb_prune_branch")


def gb_pool_set_capacity(pool: int, capacity: int) -> None:
    _check(pool, load().gb_pool_set_capacity(pool, int(capacity)), "gb_pool_set_capacity")


def gb_pool_last_ranked(pool: int, slot_out, stream=None) -> None:
    _check(pool, load().gb_pool_last_ranked(pool, ptr(slot_out), stream_handle(stream)), "gb_pool_last_ranked")


class GbScorerConfig(ctypes.Structure):
    _fields_ = [("hidden_dim", ctypes.c_int), ("ffn_dim", ctypes.c_int)]


def gb_fork_slots(pool: int, parent_of, stream=None) -> None:
    _check(pool, load().gb_fork_slots(pool, ptr(parent_of), stream_handle(stream)), "gb_fork_slots")


def gb_scorer_sizes(pool: int, cfg: GbScorerConfig, max_offsets: int = 4096):
    """(weight_bytes, workspace_bytes, [offset of each weight tensor])."""
    wb, wsb, n = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_int()
    offs = (ctypes.c_size_t * max_offsets)()
    _check(pool, load().gb_scorer_sizes(pool, ctypes.byref(cfg), ctypes.byref(wb), ctypes.byref(wsb), offs,
                                        max_offsets, ctypes.byref(n)), "gb_scorer_sizes")
    return wb.value, wsb.value, list(offs[: n.value])


def gb_scorer_seed(pool: int, cfg: GbScorerConfig, weights, workspace, h0, n_beams: int, stream=None) -> None:
    _check(pool, load().gb_scorer_seed(pool, ctypes.byref(cfg), ptr(weights), ptr(workspace), ptr(h0), n_beams,
                                       stream_handle(stream)), "gb_scorer_seed")


def gb_scorer_step(pool: int, cfg: GbScorerConfig, weights, workspace, hidden, score_out, stream=None) -> None:
    _check(pool, load().gb_scorer_step(pool, ctypes.byref(cfg), ptr(weights), ptr(workspace), ptr(hidden),
                                       ptr(score_out), stream_handle(stream)), "gb_scorer_step")


def gb_release(pool: int, slots, n: int, stream=None) -> None:
    _check(pool, load().gb_release(pool, ptr(slots), n, stream_handle(stream)), "gb_release")


def gb_pool_status(pool: int, stream=None) -> int:
    st = ctypes.c_int()
    _check(pool, load().gb_pool_status(pool, ctypes.byref(st), stream_handle(stream)), "gb_pool_status")
    return st.value


def gb_pool_clear_status(pool: int, stream=None) -> None:
    _check(pool, load().gb_pool_clear_status(pool, stream_handle(stream)), "gb_pool_clear_status")


def gb_pool_wait_selftest(pool: int, stream=None) -> None:
    _check(pool, load().gb_pool_wait_selftest(pool, stream_handle(stream)), "gb_pool_wait_selftest")


def gb_pool_read_state(pool: int, state: GbPoolState, stream=None) -> None:
    _check(pool, load().gb_pool_read_state(pool, ctypes.byref(state), stream_handle(stream)), "gb_pool_read_state")


def gb_pool_set_profile_events(pool: int, which: int, start_event=None, stop_event=None) -> None:
    """Events may be torch.cuda.Event objects (already recorded once) or raw cudaEvent_t ints."""
    def ev(e):
        if e is None or isinstance(e, int):
            return e
        return e.cuda_event
    _check(pool, load().gb_pool_set_profile_events(pool, which, ev(start_event), ev(stop_event)),
           "gb_pool_set_profile_events")


STEP_STATS_FIELDS = ("tokens_per_beam_path", "tokens_with_grouped", "seg_rowtok", "seg_tiletok", "segments",
                     "tiles", "appended", "step")


def gb_pool_read_step_stats(pool: int, max_steps: int = 4096, stream=None):
    """Work records of the last steps: an int32 array [n][10] (see include/gambit.h)."""
    import numpy as np
    out = np.zeros((max_steps, STATS_WORDS), dtype=np.int32)
    n = ctypes.c_int()
    _check(pool, load().gb_pool_read_step_stats(pool, out.ctypes.data, max_steps, ctypes.byref(n),
                                                stream_handle(stream)), "gb_pool_read_step_stats")
    return out[:n.value]


def gb_pool_launch_count(pool: int) -> int:
    n = ctypes.c_uint64()
    _check(pool, load().gb_pool_launch_count(pool, ctypes.byref(n)), "gb_pool_launch_count")
    return n.value


def gb_paged_decode_noalloc(args: GbPagedDecodeArgs, stream=None) -> None:
    """Paged decode attention with the library's fixed scratch (no allocation, no workspace)."""
    _check(None, load().gb_paged_decode_noalloc(ctypes.byref(args), stream_handle(stream)),
           "gb_paged_decode_noalloc")


def gb_paged_decode_noalloc_status(stream=None) -> int:
    """Device status of the last gb_paged_decode_noalloc call on the current device (synchronises)."""
    st = ctypes.c_int()
    _check(None, load().gb_paged_decode_noalloc_status(ctypes.byref(st), stream_handle(stream)),
           "gb_paged_decode_noalloc_status")
    return st.value


def gb_last_error(pool: int) -> str:
    return (load().gb_last_error(pool) or b"").decode()
