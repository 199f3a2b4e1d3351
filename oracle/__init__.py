"""CPU oracle of the AGN hot path.  TEST INFRASTRUCTURE ONLY: imported by the
tests, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py`, never
by the library."""
from .agn_oracle import *  # noqa: F401,F403
from .agn_oracle import __all__  # noqa: F401
