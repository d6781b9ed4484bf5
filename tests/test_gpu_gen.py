"""The device-side generator produces exactly the host generator's values (it only serves inputs)."""
import numpy as np
import pytest

from workload import gen

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_device_generator_matches_host(cuda, dtype):
    import torch
    from workload import gpu_gen
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    hs = gen.head_scales(0, 3, 4, 0.5, 2.0)
    out = torch.empty(5, 7, 4 * 16, dtype=tdt, device=cuda)
    gpu_gen.normal(out, dtype, 5, 7, 64, [11, gen.TAG_KV_K, 3, (0, 0, 1), (100, 1, 0)],
                   row_scale=torch.from_numpy(hs).to(cuda), row_scale_div=16)
    slots = np.arange(7, dtype=np.uint64)[None, :]
    pos = np.arange(100, 105, dtype=np.uint64)[:, None]
    ref = gen.kv_rows(11, gen.TAG_KV_K, 3, slots, pos, 4, 16, dtype, hs).reshape(5, 7, 64)
    got = out.float().cpu().numpy()
    assert np.array_equal(got.view(np.uint32), ref.astype(np.float32).view(np.uint32))


def test_device_generator_scaled_and_prompt_writer(cuda):
    import torch
    from workload import gpu_gen
    out = torch.empty(3, 1, 32, dtype=torch.float32, device=cuda)
    gpu_gen.normal(out, "f32", 3, 1, 32, [0, gen.TAG_KV_V, 0, gen.PROMPT_WRITER, (0, 1, 0)], scale=0.125)
    ref = gen.normal([0, gen.TAG_KV_V, 0, gen.PROMPT_WRITER, np.arange(3)], 32, 0.125)
    assert np.array_equal(out.cpu().numpy()[:, 0], ref)
