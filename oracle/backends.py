"""The oracle's two implementations behind one interface.

``"cpp"`` is the C++ oracle (``oracle/cpp/gambit_oracle.cpp``, loaded through ``oracle.cpp``):
the oracle the parity tests use.  ``"numpy"`` is the same definitions written a second time in
numpy (``oracle.attention``, ``oracle.probe``, ``oracle.tournament``, ``oracle.pool``,
``oracle.beams``); the oracle tests check the two against each other and pin both.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

from types import SimpleNamespace

NAMES = ("cpp", "numpy")
DEFAULT = "cpp"


def get(name: str = DEFAULT) -> SimpleNamespace:
    if name == "cpp":
        from oracle import cpp
        cpp.load()
        return SimpleNamespace(name="cpp", decode_attention=cpp.decode_attention,
                               softmax_weights=cpp.softmax_weights, probe_score=cpp.probe_score,
                               running_mean_update=cpp.running_mean_update, tournament=cpp.tournament,
                               rank_order=cpp.rank_order, Pool=cpp.CppPool, BeamKV=cpp.CppBeamKV)
    if name == "numpy":
        from oracle import attention, beams, pool, probe, tournament
        return SimpleNamespace(name="numpy", decode_attention=attention.decode_attention,
                               softmax_weights=attention.softmax_weights, probe_score=probe.probe_score,
                               running_mean_update=probe.running_mean_update, tournament=tournament.tournament,
                               rank_order=tournament.rank_order, Pool=pool.PoolOracle, BeamKV=beams.BeamKV)
    raise ValueError(f"unknown oracle backend {name!r}")
