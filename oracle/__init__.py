"""Plain, slow, fp64 CPU oracle of the rolling action-expert step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference leg may import it.  The CUDA library
(``paper_2609_34170_gb300``) never imports, links or calls anything here, and
nothing here imports the library: the two share no code.  Inputs come from the
seeded generators in ``synth``, which hold none of the step's arithmetic.

Modules:
  noise   -- Philox4x32-10 and the float32 Box-Muller of the appended slot
             (Sec. 3.1: the new slot is drawn from N(0, I)).
  expert  -- the action expert v_theta and the rolling update (Eq. 1, Eq. 3,
             the release / shift / append after Eq. 3, App. A.1 offsets).

Pins (tests/test_oracle_*.py, run with -m "not gpu"): Philox known-answer
vectors, own ln / sincos against libm, Euler closed forms, the single-target
ideal field, the per-action dt invariant, slot-isolated equivalence,
permutation equivariance, GQA head mapping, residual structure, brute-force
attention.  The network as a whole has no printed values in the paper: beyond
those pins its parity is "unpinned" in the sense that only its parts and their
composition laws are pinned.
"""
from . import noise, expert  # noqa: F401
