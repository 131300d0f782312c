"""Rift hot path on GB300 (sm_103a): query-conditioned tile pruning and elastic, per-tile
token-budgeted prefill.  The computation lives in libriftgb.so (C ABI: include/rift.h);
``abi`` is its ctypes binding (importing it loads the library and raises if it is missing)
and ``pipeline`` sequences the calls for one scene query.  ``build`` compiles the library."""


def __getattr__(name):
    if name in ("DeviceModel", "ScenePipeline", "interleave_gate_up"):
        from . import pipeline
        return getattr(pipeline, name)
    raise AttributeError(name)
