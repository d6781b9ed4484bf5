"""The sequence scorer (Appendix Eq. 4-6) on the device against the oracle's fp64
definition, over a search: the step pool is seeded with the prompt's hidden state,
every step scores all running traces, and forks (a tournament decided elsewhere) and
releases change which history each slot holds.

Every score the device returns is checked against ``oracle.seqscorer.seq_scores`` of
the history the slot held at that step (by causality, position t of a longer history
gives the same score, so each history that ends - by release, by being overwritten by
a fork, or at the end - is scored once and checked at every recorded position).  The
step pool's pages are compared bit for bit with ``oracle.pool.PoolOracle`` replaying
the same seed, steps, forks and releases.

Tolerance: |device - oracle| <= 8e-3 on the score, twice the bf16 bound: the device
rounds to bf16 the operands of every product (LayerNorm outputs, q/k/v, attention and
SwiGLU outputs); replaying exactly those roundings in numpy against the fp64 oracle gives
at most 4.1e-3 over 18 seeded shapes of 30 positions, and fp32 accumulation adds far less.
"""
import numpy as np
import pytest

from oracle.pool import PoolOracle
from oracle.seqscorer import SeqScorerWeights, seq_scores
from tests.parity import assert_pool_equal
from workload.scorer_weights import _bf16, seqscorer_weights

pytestmark = pytest.mark.gpu

ATOL = 8e-3


def _oracle_weights(w: dict) -> SeqScorerWeights:
    return SeqScorerWeights(w["ln_in"], w["w_in"], w["layers"], w["ln_out"], w["w_out"], w["b_out"],
                            w["n_q_heads"], w["n_kv_heads"])


@pytest.mark.parametrize("C,H,F,L,Hq,Hkv,steps,P", [
    (8, 256, 1024, 2, 4, 2, 20, 16),      # G = 2, tail pages forked mid-page
    (40, 512, 512, 1, 2, 1, 36, 16),      # two full pages shared by forked traces (grouped path)
    (130, 4096, 1024, 2, 4, 2, 6, 16),    # a ragged 128-row tile, the generator's hidden size
    (24, 256, 256, 2, 8, 2, 18, 32),      # G = 4
])
def test_scorer_matches_oracle_over_forks_and_releases(cuda, C, H, F, L, Hq, Hkv, steps, P):
    import torch
    from paper_2608_08020_gb300.seqscorer import SeqScorer
    rng = np.random.default_rng(C * 7 + H)
    w = seqscorer_weights(C + L, H, Hq * 128, F, L, Hq, Hkv)
    ow = _oracle_weights(w)
    sc = SeqScorer(w, hidden_dim=H, ffn_dim=F, max_beams=C, max_steps=steps + 1, page_size=P)
    pages_per_beam = -(-(steps + 2) // P)
    ref_pool = PoolOracle(sc.pool.num_pages, C, pages_per_beam, P)

    h0 = _bf16(rng.standard_normal(H).astype(np.float32) * 2)
    n0 = C - 3
    sc.seed(torch.from_numpy(h0).to(torch.bfloat16).cuda(), n0)
    ref_pool.seed(n0, 1)
    rows = {(-1, -1): h0}                   # hidden state of step t, slot b
    hist = {b: [(-1, -1)] for b in range(n0)}
    recorded = []                           # (history, device score)
    ended = []                              # histories that stopped growing
    score = torch.zeros(C, dtype=torch.float32, device="cuda")

    for t in range(1, steps + 1):
        hid = _bf16(rng.standard_normal((C, H)).astype(np.float32) * 2)
        sc.step(torch.from_numpy(hid).to(torch.bfloat16).cuda(), score)
        assert ref_pool.begin_step()
        got = score.cpu().numpy()
        for b in range(C):
            if b in hist:
                rows[(t, b)] = hid[b]
                hist[b].append((t, b))
                recorded.append((tuple(hist[b]), float(got[b])))
            else:
                assert got[b] == 0.0, (t, b)
        if t % 4 == 2:                      # a tournament decided on another pool
            live = sorted(hist)
            n_child = min(len(live) // 3, 6)
            parents = [int(x) for x in rng.choice(live, size=n_child, replace=True)]
            pool_of_children = [s for s in range(C) if s not in set(parents)]
            children = sorted(int(x) for x in rng.choice(pool_of_children, size=n_child, replace=False))
            parent_of = np.array([b if b in hist else -1 for b in range(C)], dtype=np.int32)
            for c, p in zip(children, parents):
                parent_of[c] = p
            sc.fork(torch.from_numpy(parent_of).cuda())
            ref_pool.fork_slots(parent_of)
            for c, p in zip(children, parents):
                if c in hist:
                    ended.append(tuple(hist[c]))
            for c, p in zip(children, parents):
                hist[c] = list(hist[p])
        if t % 5 == 3:                      # a trace completes
            s = int(rng.choice(sorted(hist)))
            ended.append(tuple(hist.pop(s)))
            sc.release(torch.tensor([s], dtype=torch.int32, device="cuda"))
            ref_pool.release([s])
    ended += [tuple(h) for h in hist.values()]

    st = sc.pool.read_state()
    assert sc.pool.status() == 0
    assert_pool_equal(st, ref_pool, P, means="exact")

    checked = set()
    worst = 0.0
    by_end = {}
    for h in ended:
        by_end.setdefault(h, None)
    for h in by_end:
        ref = seq_scores(np.stack([rows[i] for i in h]), ow)
        for rh, g in recorded:
            if len(rh) <= len(h) and h[:len(rh)] == rh and (rh, g) not in checked:
                err = abs(g - ref[len(rh) - 1])
                worst = max(worst, err)
                assert err <= ATOL, f"score of history {rh[-1]} (length {len(rh)}): device {g} oracle {ref[len(rh) - 1]}"
                checked.add((rh, g))
    assert len(checked) == len(set(recorded))
    print(f"C={C} H={H} worst score error {worst:.2e} over {len(checked)} scores")


def test_scorer_rejects_what_it_cannot_run(cuda):
    import torch
    from paper_2608_08020_gb300 import binding as B
    from paper_2608_08020_gb300.pool import BeamPool
    f32pool = BeamPool(num_layers=1, num_q_heads=2, num_kv_heads=1, head_dim=64, page_size=16, kv_dtype="f32",
                       num_pages=16, max_beams=4, max_pages_per_beam=4)
    with pytest.raises(B.GambitError):
        B.gb_scorer_sizes(f32pool.handle, B.GbScorerConfig(256, 256))
    pool = BeamPool(num_layers=1, num_q_heads=2, num_kv_heads=1, head_dim=128, page_size=16, kv_dtype="bf16",
                    num_pages=16, max_beams=4, max_pages_per_beam=4)
    with pytest.raises(B.GambitError):
        B.gb_scorer_sizes(pool.handle, B.GbScorerConfig(100, 256))       # H not a multiple of 64
    wb, wsb, offs = B.gb_scorer_sizes(pool.handle, B.GbScorerConfig(256, 256))
    assert len(offs) == 3 + 8 + 4 and all(o % 256 == 0 for o in offs) and wb > offs[-1]
    wbuf = torch.zeros(wb, dtype=torch.uint8, device="cuda")
    ws = torch.zeros(wsb, dtype=torch.uint8, device="cuda")
    h = torch.zeros((4, 256), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(4, dtype=torch.float32, device="cuda")
    with pytest.raises(B.GambitError):                                  # not seeded
        B.gb_scorer_step(pool.handle, B.GbScorerConfig(256, 256), wbuf, ws, h, out)
    assert pool.status() == 0
