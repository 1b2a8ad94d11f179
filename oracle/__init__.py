"""fp64 CPU oracle of the CRVQ code-search path. Test infrastructure only: imported by
tests/, __graft_entry__.smoke() and the CPU-baseline leg of bench.py, never by the library."""
from .crvq_oracle import *  # noqa: F401,F403
