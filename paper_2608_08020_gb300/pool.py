"""``BeamPool``: a paged beam pool whose device memory PyTorch owns.

PyTorch provides the two device buffers and the streams; every operation is
one call into ``libgambit.so`` through ``binding``.  There is no CPU path.
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_08020_gb300 import binding as B

_DT = {"f32": B.GB_F32, "bf16": B.GB_BF16}
TORCH_DT = {"f32": torch.float32, "bf16": torch.bfloat16}


class BeamPool:
    def __init__(self, *, num_layers: int, num_q_heads: int, num_kv_heads: int, head_dim: int, page_size: int,
                 kv_dtype: str, num_pages: int, max_beams: int, max_pages_per_beam: int, group_min_beams: int = 0,
                 device: str | torch.device = "cuda", stream=None):
        self.cfg = B.GbPoolConfig(num_layers, num_q_heads, num_kv_heads, head_dim, page_size, _DT[kv_dtype],
                                  num_pages, max_beams, max_pages_per_beam, group_min_beams)
        self.kv_dtype = kv_dtype
        self.max_beams = max_beams
        self.max_pages = max_pages_per_beam
        self.num_pages = num_pages
        self.device = torch.device(device)
        kv_bytes, meta_bytes = B.gb_pool_workspace_bytes(self.cfg)
        self.kv = torch.empty(kv_bytes, dtype=torch.uint8, device=self.device)
        self.meta = torch.empty(meta_bytes, dtype=torch.uint8, device=self.device)
        self.handle = B.gb_pool_init(self.cfg, self.kv, self.meta, stream)

    @classmethod
    def for_workload(cls, wl, device="cuda", num_pages: int | None = None, group_min_beams: int = 0, max_beams=None,
                     max_context: int | None = None):
        return cls(num_layers=wl.num_layers, num_q_heads=wl.num_q_heads, num_kv_heads=wl.num_kv_heads,
                   head_dim=wl.head_dim, page_size=wl.page_size, kv_dtype=wl.kv_dtype,
                   num_pages=num_pages if num_pages is not None else wl.pool_pages(max_context),
                   max_beams=max_beams if max_beams is not None else wl.beams,
                   max_pages_per_beam=wl.table_width(max_context), group_min_beams=group_min_beams, device=device)

    def close(self) -> None:
        if self.handle:
            B.gb_pool_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- operations (same names as the C ABI, minus the prefix) ---------------
    def seed(self, n_beams, prompt_len, k_prompt, v_prompt, stream=None):
        B.gb_pool_seed(self.handle, n_beams, prompt_len, k_prompt, v_prompt, stream)

    def decode_attention(self, layer, q, k_new, v_new, scale, out, flags=B.GB_PATH_AUTO, stream=None):
        B.gb_decode_attention(self.handle, layer, q, k_new, v_new, scale, out, flags, stream)

    def append_kv(self, layer, n_tokens, k, v, stream=None):
        B.gb_append_kv(self.handle, layer, n_tokens, k, v, stream)

    def score_probe(self, hidden, hidden_dtype: str, w, bias=0.0, mask=None, score_out=None, stream=None):
        B.gb_score_probe(self.handle, hidden, _DT[hidden_dtype], hidden.shape[-1], w, bias, mask, score_out, stream)

    def score_mlp(self, hidden, w1, b1, w2, b2=0.0, mask=None, score_out=None, stream=None):
        B.gb_score_mlp(self.handle, hidden, hidden.shape[-1], w1, b1, w2, b2, w1.shape[0], mask, score_out, stream)

    def push_scores(self, scores, mask=None, stream=None):
        B.gb_push_scores(self.handle, scores, mask, stream)

    def prune_branch(self, K, fanout, warmup=0, eligible=None, parent_out=None, pruned_out=None, lineage_out=None,
                     stream=None):
        B.gb_prune_branch(self.handle, K, fanout, warmup, eligible, parent_out, pruned_out, lineage_out, stream)

    def set_capacity(self, capacity: int):
        B.gb_pool_set_capacity(self.handle, capacity)

    def last_ranked(self, out, stream=None):
        """The active slot the tournament ranks last, written to the int32 device tensor `out` (-1: none)."""
        B.gb_pool_last_ranked(self.handle, out, stream)

    def release(self, slots, stream=None):
        B.gb_release(self.handle, slots, int(slots.numel()), stream)

    def status(self, stream=None) -> int:
        return B.gb_pool_status(self.handle, stream)

    def clear_status(self, stream=None):
        B.gb_pool_clear_status(self.handle, stream)

    def read_state(self, stream=None) -> dict:
        """Host copies of tables, lengths, scores, refcounts and the free bitmap."""
        C, MP, NP = self.max_beams, self.max_pages, self.num_pages
        out = {
            "tables": np.zeros((C, MP), np.int32), "seq_len": np.zeros(C, np.int32),
            "active": np.zeros(C, np.int32), "gen": np.zeros(C, np.int32), "nsteps": np.zeros(C, np.int32),
            "mean": np.zeros(C, np.float32), "lineage": np.zeros(C, np.uint32),
            "refcnt": np.zeros(NP, np.int32), "free_bits": np.zeros((NP + 31) // 32, np.uint32),
            "seg_cover": np.zeros(C, np.int32), "seg_nseg": np.zeros(C, np.int32),
        }
        st = B.GbPoolState(*[out[k].ctypes.data for k in ("tables", "seq_len", "active", "gen", "nsteps", "mean",
                                                         "lineage", "refcnt", "free_bits", "seg_cover",
                                                         "seg_nseg")])
        B.gb_pool_read_state(self.handle, st, stream)
        return out
