"""CPU oracle for the E2S-Pruner pruning decision -- TEST INFRASTRUCTURE ONLY.

A plain, slow, float64 restatement of the paper's definitions, written to
check the CUDA path.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.
The library path never calls it: there is no CPU fallback.

It shares no code with the CUDA path (no kernels, headers, helpers or
tables); both sides only consume the same seeded synthetic inputs.

Modules:
  e2s_oracle  -- Sec. 3.1 Eq. 1, Sec. 4.1-4.3 Eqs. 8-23 and Algorithm 1,
                 one function per step, in the paper's order and notation.
  ds_generic  -- the generic Dempster-Shafer definitions of Sec. 3.2
                 (Eqs. 2-7) over an arbitrary finite frame, by brute-force
                 enumeration of focal sets; used only to pin e2s_oracle.

Parity status: every step function is pinned by tests under
``tests/test_oracle_*.py`` (closed forms, the paper's worked examples,
brute force, invariants).  The whole pipeline has no printed output in the
paper to compare with, so end-to-end it is pinned only through its steps.
"""
from . import ds_generic, e2s_oracle  # noqa: F401
