"""rift_score_tiles_noalloc, the scoring entry point for callers that cannot allocate device
memory (programs whose device memory is fixed before they start, plug-ins without an allocator).
It takes its scratch from an array compiled into the library; its results must match
rift_score_tiles, which uses a caller-provided workspace, call after call.

This file is collected last on purpose: it runs after every other test, and alone.
"""
import pytest
import torch

from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _scene(wl, device):
    sc = W.make_scene(wl.scene, wl.decoder.vocab, device)
    return sc


def _outputs(wl, device):
    s = wl.scene
    f32 = dict(dtype=torch.float32, device=device)
    m = min(wl.knn_m, s.N - 1)
    return dict(r=torch.full((s.N, s.n_v), float("nan"), **f32), s0=torch.full((s.N,), float("nan"), **f32),
                s1=torch.full((s.N,), float("nan"), **f32),
                nbr=torch.full((max(s.N * m, 1),), -7, dtype=torch.int32, device=device))


def _query(abi, sc, wl, device):
    s = wl.scene
    i32 = dict(dtype=torch.int32, device=device)
    t = torch.empty(s.d, dtype=torch.float32, device=device)
    B = torch.empty(s.M, s.d, dtype=torch.float32, device=device)
    abi.query_prep(sc.embed, wl.decoder.vocab, s.d, torch.tensor(sc.query_ids, **i32), 1, s.Q,
                   torch.tensor(sc.bg_ids, **i32), s.M, t, B)
    return t, B


def _score_both(abi, wl, sc, device):
    s = wl.scene
    xdt = abi.RIFT_BF16 if s.x_dtype == "bf16" else abi.RIFT_F32
    t, B = _query(abi, sc, wl, device)
    ref, got = _outputs(wl, device), _outputs(wl, device)
    need = abi.score_workspace_bytes(s.N, s.n_v, s.d, s.M)
    ws = torch.empty(need, dtype=torch.uint8, device=device)
    abi.score_tiles(sc.X, xdt, s.N, s.n_v, s.d, t, B, s.M, wl.knn_m, ref["r"], ref["s0"], ref["s1"], ref["nbr"],
                    ws, need)
    abi.score_tiles_noalloc(sc.X, xdt, s.N, s.n_v, s.d, t, B, s.M, wl.knn_m, got["r"], got["s0"], got["s1"],
                            got["nbr"])
    abi.sync_status()
    return ref, got


def _check(ref, got):
    assert P.rel_err_rows(got["r"].cpu().numpy(), ref["r"].cpu().numpy()) < P.SCORE_RTOL
    assert P.max_abs_rel(got["s0"].cpu(), ref["s0"].cpu()) < P.SCORE_RTOL
    assert P.max_abs_rel(got["s1"].cpu(), ref["s1"].cpu()) < P.SCORE_RTOL
    assert torch.equal(got["nbr"].cpu(), ref["nbr"].cpu())


def test_noalloc_scoring_matches_workspace_scoring_twice_in_a_row(cuda, riftlib):
    # Two different scenes back to back: the second call must not see the first call's scratch.
    wl_a = W.Workload("noalloc_a", W.SceneSpec(N=64, d=4096, x_dtype="bf16"), W.LLAVA7B, W.RIFT_POLICY)
    wl_b = P.SMALL24
    for wl in (wl_a, wl_b):
        sc = _scene(wl, cuda)
        ref, got = _score_both(riftlib, wl, sc, cuda)
        _check(ref, got)


def test_noalloc_tensor_core_gram_branch_twice_in_a_row(cuda, riftlib):
    # 1100 tiles: the kNN's Gram product over its largest scene that fits the array (at d = 256),
    # with its split operands, tensor maps, split-K partials and the Gram matrix itself all inside
    # the fixed array.
    wl = W.Workload("noalloc_gram", W.SceneSpec(N=1100, d=256, x_dtype="bf16"), W.LLAVA7B, W.RIFT_POLICY)
    s = wl.scene
    assert riftlib.score_workspace_bytes(s.N, s.n_v, s.d, s.M) <= riftlib.NOALLOC_SCORE_SCRATCH_BYTES
    sc = _scene(wl, cuda)
    for _ in range(2):
        ref, got = _score_both(riftlib, wl, sc, cuda)
        _check(ref, got)


def test_noalloc_rejects_scenes_larger_than_its_array(cuda, riftlib):
    N, n_v, d, M = 2000, 576, 4096, 8
    assert riftlib.score_workspace_bytes(N, n_v, d, M) > riftlib.NOALLOC_SCORE_SCRATCH_BYTES
    x = torch.empty(16, dtype=torch.bfloat16, device=cuda)
    f = torch.empty(16, dtype=torch.float32, device=cuda)
    status = riftlib.lib.rift_score_tiles_noalloc(x.data_ptr(), riftlib.RIFT_BF16, N, n_v, d, f.data_ptr(),
                                                  f.data_ptr(), M, 6, f.data_ptr(), f.data_ptr(), f.data_ptr(),
                                                  None, 0)
    assert status == riftlib.RIFT_ERR_CAPACITY
