"""CPU oracle of the MSD decode step (arXiv 2505.14260).

TEST INFRASTRUCTURE ONLY: only tests/, __graft_entry__.smoke() and the bench's
cpu_baseline / --impl reference legs may import it. The product path (the CUDA
library and its Python binding) never imports, links or executes anything here,
and this package shares no code with it.

Every function is pinned by the tests in tests/test_oracle_pins.py; none is
"parity unpinned".
"""
from .msd_oracle import *  # noqa: F401,F403
