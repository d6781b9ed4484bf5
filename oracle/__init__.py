"""CPU oracle for the Gambit beam-decode hot path (test infrastructure only).

This package is the plain, slow, obviously correct statement of what the CUDA
library computes.  It is test infrastructure: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline / reference legs of
``bench.py`` may import it.  The product path (``paper_2608_08020_gb300``)
never imports it and shares no code with it; the only module both sides use
is the seeded input generator in ``workload/gen.py``, which holds none of the
method's arithmetic.

Modules
-------
* ``cpp/gambit_oracle.cpp`` - the oracle of the hot path in plain C++17 (attention,
  probe, running mean, tournament, the pool, beam KV copied on fork), built by
  ``build_cpp`` and loaded through ``cpp``; ``backends`` selects it (the default) or
  its numpy twin below, and the oracle tests pin both and check one against the other.
* ``attention``  - decode attention as its textbook definition (fp64,
  two-pass softmax) over each beam's full, materialised KV.
* ``probe``      - scorer probe sigma(w.h + b) in fp64 and the running-mean
  update of Algorithm 1 (the "Generate" phase) in fp32.
* ``tournament`` - the ranking and Case 1 / Case 2 routing of the
  Tournament function (Algorithm 1; Eq. 2 and Eq. 3).
* ``pool``       - the paged pool as plain Python state: per-slot block
  tables, page refcounts, lowest-free-page allocation, copy-on-write of a
  shared partial tail page, and each beam's writer history.
* ``beams``      - a literal copy-on-fork model that keeps every beam's full
  K/V arrays (copying the parent's arrays when a child is branched), and
  the same KV rebuilt from the writer history for large sampled checks.
* ``simulate``   - the main loop of Algorithm 1 with trace completion, used
  to pin the tournament's node accounting against the paper's runtime example.

Parity pins: every function here is checked by ``tests/test_oracle_*.py``
against closed forms, invariants, brute force and the paper's printed
accounting, never against the CUDA path.
"""
