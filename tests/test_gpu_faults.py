"""Failure paths on the GPU, injected from the host (no fault, trap or hang of the GPU): a bounded
wait that runs out, corrupted selections and ids, and capacities that are too small.  Each sets a
device flag that rift_sync_status returns, and the context stays usable."""
from dataclasses import replace

import pytest
import torch

from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _status(riftlib):
    return riftlib.lib.rift_sync_status(None)


def test_a_wait_that_never_completes_gives_up_with_a_timeout(cuda, riftlib):
    assert _status(riftlib) == riftlib.RIFT_OK
    riftlib.check_wait_timeout()
    assert _status(riftlib) == riftlib.RIFT_ERR_TIMEOUT
    # the context still works: a real product afterwards is right
    a = torch.randn(64, 128, device=cuda).half()
    w = torch.randn(96, 128, device=cuda).half()
    out = torch.empty(64, 96, dtype=torch.float16, device=cuda)
    riftlib.linear(a, w, 64, 96, 128, riftlib.RIFT_EPI_STORE_F16, out)
    assert _status(riftlib) == riftlib.RIFT_OK
    ref = a.float() @ w.float().T
    assert float((out.float() - ref).abs().max() / ref.abs().max()) < 2e-3


def _selected(wl, cuda):
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    pipe.select(dv["X"], dv["embed"], dv["q"], dv["bg"])
    return sc, pipe, dv


def test_pack_flags_corrupted_selection_and_ids(cuda, riftlib):
    wl = P.SMALL24
    sc, pipe, dv = _selected(wl, cuda)
    assert _status(riftlib) == riftlib.RIFT_OK
    pipe.sel[0] = wl.scene.n_v + 5                      # a token index past the tile
    pipe.pack(dv["X"], dv["embed"], dv["sys"], dv["q"])
    assert _status(riftlib) == riftlib.RIFT_ERR_BAD_ID
    pipe.select(dv["X"], dv["embed"], dv["q"], dv["bg"])   # a clean selection again
    bad_q = dv["q"].clone()
    bad_q[1] = sc.embed.shape[0]                         # a query id past the vocabulary
    pipe.pack(dv["X"], dv["embed"], dv["sys"], bad_q)
    assert _status(riftlib) == riftlib.RIFT_ERR_BAD_ID
    pipe.pack(dv["X"], dv["embed"], dv["sys"], dv["q"])
    assert _status(riftlib) == riftlib.RIFT_OK


def test_merge_capacity_overflow_writes_no_contextual_rows(cuda, riftlib):
    wl = replace(P.SMALL24, policy=replace(P.SMALL24.policy, ctx_num=10, ctx_den=64))
    sc, pipe, dv = _selected(wl, cuda)
    pipe.max_ctx = 1                                     # far below the tiles' contextual tokens
    pipe.merge(dv["X"])
    assert _status(riftlib) == riftlib.RIFT_ERR_CAPACITY
    n = int(pipe.n_kept.item())
    assert pipe.ctx_off[:n + 1].cpu().tolist() == [0] * (n + 1)
