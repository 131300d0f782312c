"""CPU oracle for the Rift hot path.  Test infrastructure only: imported by tests/,
__graft_entry__.smoke() and bench.py's CPU-baseline leg, never by the library."""
from .rift_oracle import *  # noqa: F401,F403
