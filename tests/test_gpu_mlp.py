"""The two-layer MLP scorer on the tensor cores (gb_score_mlp) against the oracle's fp64
sigma(w2 . relu(W1 h + b1) + b2): partial row and column tiles, several K splits, inactive
slots, the boundary mask and the running-mean update."""
import numpy as np
import pytest

from oracle.probe import mlp_probe_score, running_mean_update
from tests.parity import assert_close

pytestmark = pytest.mark.gpu


def _bf16(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest even) and back, as the device sees the values."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return u.astype(np.uint32).view(np.float32)


@pytest.mark.parametrize("C,H,dh", [(8, 256, 128), (200, 4096, 200), (512, 4096, 512), (64, 1024, 40)])
def test_mlp_scores_and_means_match_oracle(cuda, C, H, dh):
    import torch
    from paper_2608_08020_gb300.pool import BeamPool
    rng = np.random.default_rng(C + H + dh)
    pool = BeamPool(num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16, kv_dtype="bf16",
                    num_pages=C * 4 + 8, max_beams=C, max_pages_per_beam=4)
    kp = torch.zeros((1, 16, 8, 128), dtype=torch.bfloat16, device="cuda")
    pool.seed(C, 16, kp, kp)
    h = _bf16(rng.standard_normal((C, H)).astype(np.float32))
    w1 = _bf16((rng.standard_normal((dh, H)) / np.sqrt(H)).astype(np.float32))
    b1 = (rng.standard_normal(dh) * 0.1).astype(np.float32)
    w2 = (rng.standard_normal(dh) / np.sqrt(dh)).astype(np.float32)
    b2 = 0.1
    ref = mlp_probe_score(h, w1, b1, w2, b2)
    td = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(dt).cuda()
    score = torch.zeros(C, dtype=torch.float32, device="cuda")
    for rep in range(2):                                   # the second call sees n = 1
        pool.score_mlp(td(h, torch.bfloat16), td(w1, torch.bfloat16), td(b1, torch.float32), td(w2, torch.float32),
                       b2, score_out=score)
        got = score.cpu().numpy()
        assert_close(got, ref, "bf16", f"mlp scores C={C} H={H} d_h={dh}")
    st = pool.read_state()
    for b in range(C):                                     # the mean of two identical scores is that score
        m1, n1 = running_mean_update(np.float32(0), 0, np.float32(got[b]))
        m2, n2 = running_mean_update(m1, n1, np.float32(got[b]))
        assert st["mean"][b] == m2 and st["nsteps"][b] == n2
    assert pool.status() == 0


def test_mlp_mask_and_inactive_slots(cuda):
    import torch
    from paper_2608_08020_gb300.pool import BeamPool
    C, H, dh = 16, 128, 64
    rng = np.random.default_rng(3)
    pool = BeamPool(num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16, kv_dtype="bf16",
                    num_pages=64, max_beams=C, max_pages_per_beam=4)
    kp = torch.zeros((1, 16, 8, 128), dtype=torch.bfloat16, device="cuda")
    pool.seed(10, 16, kp, kp)                              # slots 10..15 inactive
    h = torch.from_numpy(_bf16(rng.standard_normal((C, H)).astype(np.float32))).to(torch.bfloat16).cuda()
    w1 = torch.from_numpy(_bf16(rng.standard_normal((dh, H)).astype(np.float32) / 16)).to(torch.bfloat16).cuda()
    b1 = torch.zeros(dh, dtype=torch.float32, device="cuda")
    w2 = torch.full((dh,), 0.05, dtype=torch.float32, device="cuda")
    mask = torch.tensor([1, 0] * 8, dtype=torch.uint8, device="cuda")
    score = torch.full((C,), -1.0, dtype=torch.float32, device="cuda")
    pool.score_mlp(h, w1, b1, w2, 0.0, mask=mask, score_out=score)
    s = score.cpu().numpy()
    st = pool.read_state()
    assert np.all(s[10:] == 0.0) and np.all(s[:10] > 0.0)
    assert list(st["nsteps"][:10]) == [1, 0] * 5
    assert pool.status() == 0
