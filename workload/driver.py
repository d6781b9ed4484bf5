"""Drive a workload schedule through the C ABI (``paper_2608_08020_gb300``).

Inputs come from the seeded generator: on the host (``workload.gen``, numpy)
for small cases, or on the device (``workload.gpu_gen``) for large ones; the
two produce identical values.  Inputs are keyed by (layer, writer slot,
position), so the values a slot writes depend only on where it is, and the
CPU oracle can regenerate the KV of any beam from its writer history.

All active beams of a pool advance together, so the shared context length is
tracked on the host (``self.pos``).
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_08020_gb300 import binding as B
from paper_2608_08020_gb300.pool import TORCH_DT, BeamPool
from workload import gen
from workload.configs import Workload


class GpuRun:
    def __init__(self, wl: Workload, device_gen: bool = False, device: str = "cuda", num_pages: int | None = None,
                 group_min_beams: int = 0, max_chunk: int = 256, max_context: int | None = None):
        self.wl = wl
        self.device_gen = device_gen
        self.dev = torch.device(device)
        self.pool = BeamPool.for_workload(wl, device=device, num_pages=num_pages, group_min_beams=group_min_beams,
                                          max_context=max_context)
        C, Hq, Hkv, D = wl.beams, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
        self.C = C
        self.tdt = TORCH_DT[wl.kv_dtype]
        self.q = torch.zeros(C, Hq, D, dtype=self.tdt, device=self.dev)
        self.k_new = torch.zeros(C, Hkv, D, dtype=self.tdt, device=self.dev)
        self.v_new = torch.zeros(C, Hkv, D, dtype=self.tdt, device=self.dev)
        self.out = torch.zeros(wl.num_layers, C, Hq, D, dtype=torch.float32, device=self.dev)
        self.hidden = torch.zeros(C, wl.hidden, dtype=TORCH_DT[wl.hidden_dtype], device=self.dev)
        self.scores = torch.zeros(C, dtype=torch.float32, device=self.dev)
        self.parent = torch.zeros(C, dtype=torch.int32, device=self.dev)
        self.pruned = torch.zeros(C, dtype=torch.uint8, device=self.dev)
        self.lineage = torch.zeros(C, dtype=torch.int32, device=self.dev)
        self.max_chunk = max_chunk
        self.chunk_k = None
        self.chunk_v = None
        w = gen.probe_weight(wl.seed, wl.hidden, wl.w_scale)
        self.w = torch.from_numpy(w).to(self.dev)
        self.hscale = None
        if wl.head_scale is not None:
            self.hscale = [gen.head_scales(wl.seed, l, Hkv, *wl.head_scale) for l in range(wl.num_layers)]
            self.hscale_dev = [torch.from_numpy(h).to(self.dev) for h in self.hscale]
        self.pos = 0

    # -- input generation ----------------------------------------------------
    def _host(self, x: np.ndarray, dtype) -> torch.Tensor:
        return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(self.dev).to(dtype)

    def _gen_kv(self, which: int, layer: int, pos0: int, n: int, out: torch.Tensor) -> None:
        """K or V rows for every slot at positions pos0..pos0+n-1: out [n][C][Hkv][D]."""
        wl = self.wl
        if self.device_gen:
            from workload import gpu_gen
            gpu_gen.normal(out, wl.kv_dtype, n, self.C, wl.num_kv_heads * wl.head_dim,
                           [wl.seed, which, layer, (0, 0, 1), (pos0, 1, 0)],
                           row_scale=self.hscale_dev[layer] if self.hscale else None, row_scale_div=wl.head_dim)
        else:
            slots = np.arange(self.C, dtype=np.uint64)[None, :]
            pos = np.arange(pos0, pos0 + n, dtype=np.uint64)[:, None]
            x = gen.kv_rows(wl.seed, which, layer, slots, pos, wl.num_kv_heads, wl.head_dim, wl.kv_dtype,
                            self.hscale[layer] if self.hscale else None)
            out.copy_(self._host(x, self.tdt).view_as(out))

    def _gen_q(self, layer: int, pos: int) -> None:
        wl = self.wl
        if self.device_gen:
            from workload import gpu_gen
            gpu_gen.normal(self.q, wl.kv_dtype, 1, self.C, wl.num_q_heads * wl.head_dim,
                           [wl.seed, gen.TAG_Q, layer, (0, 0, 1), pos],
                           scale=wl.q_scale if wl.q_scale is not None else 1.0)
        else:
            x = gen.q_rows(wl.seed, layer, np.arange(self.C), pos, wl.num_q_heads, wl.head_dim, wl.kv_dtype,
                           wl.q_scale)
            self.q.copy_(self._host(x, self.tdt))

    def _gen_hidden(self, pos: int) -> None:
        wl = self.wl
        if self.device_gen:
            from workload import gpu_gen
            gpu_gen.normal(self.hidden, wl.hidden_dtype, 1, self.C, wl.hidden,
                           [wl.seed, gen.TAG_HIDDEN, (0, 0, 1), pos])
        else:
            x = gen.hidden_rows(wl.seed, np.arange(self.C), pos, wl.hidden, wl.hidden_dtype)
            self.hidden.copy_(self._host(x, self.hidden.dtype))

    def prompt_kv(self) -> tuple[torch.Tensor, torch.Tensor]:
        wl = self.wl
        T = wl.prompt_len
        shape = (wl.num_layers, T, wl.num_kv_heads, wl.head_dim)
        k = torch.empty(shape, dtype=self.tdt, device=self.dev)
        v = torch.empty(shape, dtype=self.tdt, device=self.dev)
        for layer in range(wl.num_layers):
            for which, dst in ((gen.TAG_KV_K, k), (gen.TAG_KV_V, v)):
                if self.device_gen:
                    from workload import gpu_gen
                    gpu_gen.normal(dst[layer], wl.kv_dtype, T, 1, wl.num_kv_heads * wl.head_dim,
                                   [wl.seed, which, layer, gen.PROMPT_WRITER, (0, 1, 0)],
                                   row_scale=self.hscale_dev[layer] if self.hscale else None,
                                   row_scale_div=wl.head_dim)
                else:
                    x = gen.kv_rows(wl.seed, which, layer, gen.PROMPT_WRITER, np.arange(T, dtype=np.uint64),
                                    wl.num_kv_heads, wl.head_dim, wl.kv_dtype,
                                    self.hscale[layer] if self.hscale else None)
                    dst[layer].copy_(self._host(x, self.tdt))
        return k, v

    # -- schedule steps --------------------------------------------------------
    def seed(self) -> None:
        k, v = self.prompt_kv()
        self.pool.seed(self.C, self.wl.prompt_len, k, v)
        self.pos = self.wl.prompt_len

    def decode_step(self, flags: int = B.GB_PATH_AUTO) -> torch.Tensor:
        """One token for every beam and layer; returns out [layers][C][Hq][D] (device)."""
        for layer in range(self.wl.num_layers):
            self._gen_q(layer, self.pos)
            self._gen_kv(gen.TAG_KV_K, layer, self.pos, 1, self.k_new.view(1, *self.k_new.shape))
            self._gen_kv(gen.TAG_KV_V, layer, self.pos, 1, self.v_new.view(1, *self.v_new.shape))
            self.pool.decode_attention(layer, self.q, self.k_new, self.v_new, self.wl.attn_scale, self.out[layer],
                                       flags)
        self.pos += 1
        return self.out

    def append(self, n: int) -> None:
        """Append n tokens per beam (chunked), without attention."""
        wl = self.wl
        while n > 0:
            m = min(n, self.max_chunk)
            shape = (m, self.C, wl.num_kv_heads, wl.head_dim)
            if self.chunk_k is None or self.chunk_k.shape[0] < m:
                self.chunk_k = torch.empty((self.max_chunk,) + shape[1:], dtype=self.tdt, device=self.dev)
                self.chunk_v = torch.empty_like(self.chunk_k)
            ck, cv = self.chunk_k[:m], self.chunk_v[:m]
            for layer in range(wl.num_layers):
                self._gen_kv(gen.TAG_KV_K, layer, self.pos, m, ck)
                self._gen_kv(gen.TAG_KV_V, layer, self.pos, m, cv)
                self.pool.append_kv(layer, m, ck, cv)
            self.pos += m
            n -= m

    def probe(self, mask=None) -> torch.Tensor:
        self._gen_hidden(self.pos)
        self.pool.score_probe(self.hidden, self.wl.hidden_dtype, self.w, self.wl.bias, mask, self.scores)
        return self.scores

    def prune(self, K: int | None = None, fanout: int | None = None, warmup: int | None = None, eligible=None):
        wl = self.wl
        self.pool.prune_branch(wl.K if K is None else K, wl.fanout if fanout is None else fanout,
                               wl.warmup if warmup is None else warmup, eligible, self.parent, self.pruned,
                               self.lineage)
        return self.parent, self.pruned, self.lineage

    def build(self, upto: int | None = None, final_round: bool = False) -> None:
        """Seed and run the schedule (appends, probe + tournament at each round) up to length `upto`."""
        wl = self.wl
        upto = wl.context if upto is None else upto
        self.seed()
        for L in wl.rounds(include_final=final_round):
            if L > upto:
                break
            self.append(L - self.pos)
            self.probe()
            self.prune()
        if upto > self.pos:
            self.append(upto - self.pos)
