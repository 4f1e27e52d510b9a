"""CPU oracle for the DriveCache hot path (fp64 planner, fp64 DiT).

TEST INFRASTRUCTURE ONLY: only `tests/`, `__graft_entry__.smoke()` and the
benchmark's CPU-baseline leg may import it.  The product library never calls
into it and shares no code with it; both sides draw seeded inputs from
`synth` only.

Parity pins: every function is checked in `tests/test_oracle_*.py` against
closed forms, brute force, library routines and invariants.  The absolute
accuracy of a cached output relative to full inference has no pin in the
paper (it reports PSNR on real generators only): parity unpinned for that
quantity; the oracle replays the algorithm step by step instead.
"""

from . import planner, dit, controller  # noqa: F401
