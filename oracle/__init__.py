"""CPU oracle of the DensityKV hot path: TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
leg of ``bench.py`` may import this package.  It shares no code with the CUDA
library and is never on the product path.

Parity status: every function is pinned by the ``-m "not gpu"`` tests in
``tests/test_oracle_*.py`` (closed forms, identities of App. A-B, brute force
on tiny banks, the invariants of App. C, a hand-derived worked example, the
storage figures printed in App. D, and a textbook attention routine).  The
paper's end-to-end quality outcome (VBench) is not reproduced and is not a
parity target.
"""
from .densitykv import *  # noqa: F401,F403
