"""fp64 CPU oracle of the Chimera draft-and-verify step.

Test infrastructure: only tests/, `__graft_entry__.smoke()` and the benchmark's
CPU-baseline leg may import it.  The product path never does.
"""
from . import chimera_oracle, tree  # noqa: F401
