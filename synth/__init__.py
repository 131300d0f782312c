"""Seeded synthetic inputs shared by the oracle, the tests and the benchmark.  Holds none of
the method's arithmetic."""
from . import rng, workloads  # noqa: F401
