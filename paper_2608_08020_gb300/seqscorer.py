"""``SeqScorer``: the history-aware sequence scorer (Appendix, "Evaluating Search
Generalization", Eq. 4-6) on the device, one position per thought step.

The scorer's key/value cache is a second ``BeamPool`` (the step pool, one token per
thought step, bf16, 128-dim heads) whose slots mirror the generator pool's: seed it
with the prompt's final hidden state, call ``step`` at every thought boundary, and
mirror the generator's tournaments with ``fork`` (its ``parent_out``) and its
completions and evictions with ``release``.  A branched trace then continues from its
parent's scorer history without copying it, as it does for its KV.

Every operation is one call into ``libgambit.so`` (gb_scorer_*, gb_fork_slots).
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_08020_gb300 import binding as B
from paper_2608_08020_gb300.pool import BeamPool

HEAD_DIM = 128


def _bf16_bytes(a) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint8).reshape(-1)


def _f32_bytes(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32).view(np.uint8).reshape(-1)


def pack_weights(w: dict, offsets: list, total: int) -> np.ndarray:
    """Lay out the scorer's weights in the library's buffer order (gambit.h, gb_scorer_*).

    ``w``: ln_in (gain, bias), w_in [d][H], layers (each ln1, wq, wk, wv, wo, ln2, w1, w3,
    w2), ln_out, w_out [d], b_out; matrices are converted to bf16, the rest kept fp32."""
    parts = [_f32_bytes(w["ln_in"][0]), _f32_bytes(w["ln_in"][1]), _bf16_bytes(w["w_in"])]
    for L in w["layers"]:
        parts += [_f32_bytes(L["ln1"][0]), _f32_bytes(L["ln1"][1]),
                  _bf16_bytes(np.concatenate([L["wq"], L["wk"], L["wv"]], axis=0)), _bf16_bytes(L["wo"]),
                  _f32_bytes(L["ln2"][0]), _f32_bytes(L["ln2"][1]),
                  _bf16_bytes(np.concatenate([L["w1"], L["w3"]], axis=0)), _bf16_bytes(L["w2"])]
    parts += [_f32_bytes(w["ln_out"][0]), _f32_bytes(w["ln_out"][1]), _f32_bytes(w["w_out"]),
              _f32_bytes([w["b_out"]])]
    if len(parts) != len(offsets):
        raise ValueError(f"weights have {len(parts)} tensors, the library expects {len(offsets)}")
    buf = np.zeros(total, dtype=np.uint8)
    for i, (o, p) in enumerate(zip(offsets, parts)):
        end = offsets[i + 1] if i + 1 < len(offsets) else total
        if o + p.size > end:
            raise ValueError(f"weight tensor {i} has {p.size} bytes, its slot {end - o}")
        buf[o:o + p.size] = p
    return buf


class SeqScorer:
    def __init__(self, weights: dict, *, hidden_dim: int, ffn_dim: int, max_beams: int, max_steps: int,
                 page_size: int = 16, num_pages: int | None = None, device: str | torch.device = "cuda"):
        Hq, Hkv = int(weights["n_q_heads"]), int(weights["n_kv_heads"])
        pages_per_beam = -(-(max_steps + 1) // page_size)
        if num_pages is None:
            num_pages = max_beams * pages_per_beam + max_beams
        self.pool = BeamPool(num_layers=len(weights["layers"]), num_q_heads=Hq, num_kv_heads=Hkv,
                             head_dim=HEAD_DIM, page_size=page_size, kv_dtype="bf16", num_pages=num_pages,
                             max_beams=max_beams, max_pages_per_beam=pages_per_beam, device=device)
        self.cfg = B.GbScorerConfig(hidden_dim, ffn_dim)
        self.hidden_dim, self.max_beams = hidden_dim, max_beams
        wb, wsb, offs = B.gb_scorer_sizes(self.pool.handle, self.cfg)
        self.offsets = offs
        self.weights = torch.from_numpy(pack_weights(weights, offs, wb)).to(self.pool.device)
        self.workspace = torch.empty(wsb, dtype=torch.uint8, device=self.pool.device)

    def seed(self, h0: torch.Tensor, n_beams: int, stream=None) -> None:
        """Position 0 of every trace: h0 bf16 [H], the hidden state at the end of the prompt."""
        B.gb_scorer_seed(self.pool.handle, self.cfg, self.weights, self.workspace, h0, n_beams, stream)

    def step(self, hidden: torch.Tensor, score_out: torch.Tensor, stream=None) -> None:
        """One thought boundary: hidden bf16 [max_beams][H] -> score_out fp32 [max_beams] (Eq. 6)."""
        B.gb_scorer_step(self.pool.handle, self.cfg, self.weights, self.workspace, hidden, score_out, stream)

    def fork(self, parent_of: torch.Tensor, stream=None) -> None:
        """Mirror a tournament: parent_of int32 [max_beams] (gb_prune_branch's parent_out)."""
        B.gb_fork_slots(self.pool.handle, parent_of, stream)

    def release(self, slots: torch.Tensor, stream=None) -> None:
        self.pool.release(slots, stream)
