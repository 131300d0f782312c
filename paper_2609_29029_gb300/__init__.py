"""Rift hot path on GB300 (sm_103a): query-conditioned tile pruning and elastic, per-tile
token-budgeted prefill.  The computation lives in libriftgb.so (C ABI: include/rift.h);
``abi`` is its ctypes binding and ``pipeline`` sequences the calls for one scene query."""
from . import abi  # noqa: F401  (loads libriftgb.so; raises if it is missing)
from .pipeline import DeviceModel, ScenePipeline, interleave_gate_up  # noqa: F401
