"""Synthetic workloads: shapes, tree-building schedules and input recipes.

The paper measures on AIME/HMMT/GPQA traces of Qwen3-4B/8B and Phi-4 served by
vLLM (Section 4); none of those models, datasets or scorer weights are used
here.  Seeded synthetic inputs with the Qwen3-8B attention shape (32 query /
8 KV heads, head dim 128, hidden 4096, 36 layers) stand in for them, and the
beam trees are built by real prune/branch rounds driven by seeded probe
scores, with tree shapes taken from the paper (capacity C = 256, traces of
16-35K tokens, forks every Delta tokens).

A schedule is: seed ``beams`` root traces on a ``prompt_len``-token shared
prompt, then advance all beams; at every ``rounds()`` length L the probe is
evaluated once per beam (all beams at a thought boundary) and one tournament
round runs with swap size ``K`` and fan-out ``fanout``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field


@dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    kv_dtype: str            # 'f32' or 'bf16' (also the query dtype)
    beams: int               # capacity C
    prompt_len: int
    context: int             # final context length L
    interval: int            # tokens between tournament rounds
    K: int                   # swap size
    fanout: int
    hidden: int              # probe hidden size H
    hidden_dtype: str
    w_scale: float           # probe weight std (exact power of two)
    q_scale: float | None    # generator scale of q (None: unscaled N(0,1))
    attn_scale: float        # softmax scale passed to the kernel
    head_scale: tuple | None = None  # per-KV-head value scale U(lo, hi) of K and V
    bias: float = 0.0
    seed: int = 0
    num_pages: int | None = None
    pool_bytes: int | None = None    # fixed pool size (memory-capped workload)
    warmup: int = 0
    extra: dict = field(default_factory=dict)

    @property
    def G(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def esize(self) -> int:
        return 2 if self.kv_dtype == "bf16" else 4

    @property
    def pages_per_beam(self) -> int:
        return -(-self.context // self.page_size)

    def table_width(self, max_context: int | None = None) -> int:
        """Block-table entries per slot for contexts up to max_context (default: the workload's)."""
        return -(-(max_context or self.context) // self.page_size) + 1

    def kv_bytes_per_token_layer(self) -> int:
        return 2 * self.num_kv_heads * self.head_dim * self.esize

    def page_bytes_all_layers(self) -> int:
        return self.num_layers * self.page_size * self.kv_bytes_per_token_layer()

    def pool_pages(self, max_context: int | None = None) -> int:
        if self.num_pages is not None:
            return self.num_pages
        if self.pool_bytes is not None:
            return self.pool_bytes // self.page_bytes_all_layers()
        # Enough for every beam to hold its whole context unshared, plus slack.
        return self.beams * (self.table_width(max_context) + 1) + 64

    def rounds(self, include_final: bool = False) -> list[int]:
        """Context lengths at which probe + tournament run during the build."""
        out, L = [], self.prompt_len + self.interval
        while L < self.context or (include_final and L == self.context):
            out.append(L)
            L += self.interval
        return out


TINY = Workload(
    name="tiny-fp32-8beams", num_layers=1, num_q_heads=4, num_kv_heads=2, head_dim=64, page_size=16,
    kv_dtype="f32", beams=8, prompt_len=64, context=256, interval=96, K=4, fanout=2,
    hidden=256, hidden_dtype="f32", w_scale=1.0 / 16, q_scale=1.0 / 8, attn_scale=1.0)

QWEN3_8B_LAYER = Workload(
    name="qwen3-8b-layer-64beams-L4096", num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128,
    page_size=16, kv_dtype="bf16", beams=64, prompt_len=512, context=4096, interval=512, K=32, fanout=2,
    hidden=4096, hidden_dtype="bf16", w_scale=1.0 / 64, q_scale=None, attn_scale=1.0 / math.sqrt(128))

PARALLEL_SAMPLING = Workload(
    name="parallel-sampling-512beams-L16384", num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128,
    page_size=16, kv_dtype="bf16", beams=512, prompt_len=1024, context=16384, interval=1024, K=384, fanout=4,
    hidden=4096, hidden_dtype="bf16", w_scale=1.0 / 64, q_scale=None, attn_scale=1.0 / math.sqrt(128),
    head_scale=(0.5, 2.0))

LONG_CONTEXT = Workload(
    name="long-context-256beams-L32768-P32", num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128,
    page_size=32, kv_dtype="bf16", beams=256, prompt_len=4096, context=32768, interval=2048, K=128, fanout=2,
    hidden=4096, hidden_dtype="bf16", w_scale=1.0 / 64, q_scale=None, attn_scale=1.0 / math.sqrt(128))

MEMORY_CAPPED = Workload(
    name="memory-capped-36layers-L8192-120GB", num_layers=36, num_q_heads=32, num_kv_heads=8, head_dim=128,
    page_size=16, kv_dtype="bf16", beams=198, prompt_len=512, context=8192, interval=512, K=99, fanout=2,
    hidden=4096, hidden_dtype="bf16", w_scale=1.0 / 64, q_scale=None, attn_scale=1.0 / math.sqrt(128),
    pool_bytes=120 * 10**9)

# No shared KV at all: 64 independent traces of 16384 tokens (a one-token prompt, whose partly
# filled page every trace but one copies on its first append, and no tournament, so no forks).
# Every page is read by one beam only: the per-beam path's own roofline.
UNSHARED = Workload(
    name="unshared-64beams-L16384", num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128,
    page_size=16, kv_dtype="bf16", beams=64, prompt_len=1, context=16384, interval=1 << 30, K=0, fanout=2,
    hidden=4096, hidden_dtype="bf16", w_scale=1.0 / 64, q_scale=None, attn_scale=1.0 / math.sqrt(128))

ALL = {w.name: w for w in (TINY, QWEN3_8B_LAYER, PARALLEL_SAMPLING, LONG_CONTEXT, MEMORY_CAPPED, UNSHARED)}
BY_INDEX = [TINY, QWEN3_8B_LAYER, PARALLEL_SAMPLING, LONG_CONTEXT, MEMORY_CAPPED, UNSHARED]
