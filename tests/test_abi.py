"""The C-ABI library loads and exports every symbol include/gambit.h declares (no GPU needed)."""
import ctypes
import re
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parent.parent
HEADER = ROOT / "include" / "gambit.h"


def declared_functions():
    text = re.sub(r"/\*.*?\*/", "", HEADER.read_text(), flags=re.S)
    return re.findall(r"^\s*(?:gb_status|const char\s*\*)\s*(gb_\w+)\s*\(", text, flags=re.M)


def _lib():
    from paper_2608_08020_gb300 import binding
    if not binding.LIB_PATH.exists():
        pytest.skip("libgambit.so not built")
    import torch  # noqa: F401  (loads the CUDA runtime the library links against)
    return binding, binding.load()


def test_header_declares_the_hot_path_calls():
    names = declared_functions()
    for n in ("gb_pool_init", "gb_decode_attention", "gb_score_probe", "gb_prune_branch", "gb_release"):
        assert n in names


def test_every_declared_symbol_is_exported():
    binding, lib = _lib()
    names = declared_functions()
    assert sorted(names) == sorted(binding.EXPORTS)
    for n in names:
        assert hasattr(lib, n), n


def test_workspace_sizes_without_a_gpu():
    binding, _ = _lib()
    cfg = binding.GbPoolConfig(1, 32, 8, 128, 16, binding.GB_BF16, 1000, 64, 257, 0)
    kv, meta = binding.gb_pool_workspace_bytes(cfg)
    assert kv == 1 * 1000 * 2 * 8 * 16 * 128 * 2
    assert meta > 64 * 257 * 4


@pytest.mark.parametrize("bad,code", [
    (dict(num_q_heads=30), "GB_ERR_INVALID"),     # Hq not a multiple of Hkv
    (dict(page_size=24), "GB_ERR_INVALID"),
    (dict(max_beams=2048), "GB_ERR_INVALID"),
    (dict(head_dim=96), "GB_ERR_UNSUPPORTED"),
    (dict(kv_dtype=7), "GB_ERR_INVALID"),
])
def test_invalid_configs_are_rejected(bad, code):
    binding, _ = _lib()
    base = dict(num_layers=1, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16,
                kv_dtype=binding.GB_BF16, num_pages=100, max_beams=8, max_pages_per_beam=16, group_min_beams=0)
    base.update(bad)
    cfg = binding.GbPoolConfig(**base)
    with pytest.raises(binding.GambitError) as e:
        binding.gb_pool_workspace_bytes(cfg)
    assert code in str(e.value)


def test_binding_fails_loudly_without_the_library(tmp_path):
    from paper_2608_08020_gb300 import binding
    with pytest.raises(RuntimeError):
        binding.load(tmp_path / "missing.so")
