"""Degenerate scenes through the whole CUDA path against the oracle: one tile (min-max has no
spread, so u = 1 and the tile is kept; no neighbours), two tiles without background terms (Eq. 1
is the plain cosine; smoothing over the one neighbour makes both scores equal, so u = 1 for
both), no smoothing (m = 0), and nine tiles with one planted.  Then the size limits of the C ABI
(the longest tiles and the widest embeddings it accepts) and empty batches."""
from dataclasses import replace

import numpy as np
import pytest
import torch

from oracle import rift_oracle as O
from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu

BASE = W.TINY
EDGE = {
    "one_tile": replace(BASE, scene=replace(BASE.scene, N=1, planted_frac=1.0, distractor_frac=0.0)),
    "two_tiles_no_background": replace(BASE, scene=replace(BASE.scene, N=2, M=0, planted_frac=0.5,
                                                           distractor_frac=0.0)),
    "no_smoothing": replace(BASE, scene=replace(BASE.scene, N=7, planted_frac=0.3, distractor_frac=0.3), knn_m=0),
    "nine_tiles_one_planted": replace(BASE, scene=replace(BASE.scene, N=9, planted_frac=0.12, distractor_frac=0.0)),
}


def _model(dec, device):
    from paper_2609_29029_gb300 import DeviceModel
    layers = [W.make_layer(dec, l, "cpu") for l in range(dec.n_layers)]
    gf = W.make_final_norm(dec, "cpu")
    return DeviceModel(dec, layers, gf, device), layers, gf


@pytest.mark.parametrize("name", sorted(EDGE))
def test_degenerate_scene_matches_oracle(name, cuda, riftlib):
    wl = EDGE[name]
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    sel = P.oracle_select(wl, sc)
    P.assert_margins(sel, wl)
    assert len(sel.kept) >= 1  # the best tile always survives min-max and tau
    dm, layers, gf = _model(wl.decoder, cuda)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, model=dm)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"])
    riftlib.sync_status()
    r = pipe.result(n_kept, T)
    assert r.kept.cpu().tolist() == sel.kept
    assert r.budgets.cpu().tolist() == sel.budgets
    off = r.sel_off.cpu().tolist()
    got = r.sel.cpu().tolist()
    assert [got[off[j]:off[j + 1]] for j in range(n_kept)] == [list(s) for s in sel.sel]
    if wl.scene.N == 1:
        assert float(r.u.cpu()[0]) == 1.0
    H0, cu, _ = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    assert r.cu_seqlens.cpu().tolist() == list(cu)
    out = r.hidden.cpu()
    errs = [P.max_abs_rel(out[a:b], O.prefill_sequence(H0[a:b], lambda l: layers[l], gf, wl.decoder))
            for a, b in P.seq_slices(cu)]
    assert max(errs) < P.HIDDEN_TOL, errs


# The largest tile length (n_v = 1024, a 32 x 32 token grid) and width (d = 8192) the ABI takes,
# with the budget set scaled to the tile and caller-given p_i that reach the whole-tile budget.
MAX_DIMS = W.Workload("max_dims_bf16", W.SceneSpec(N=8, d=8192, x_dtype="bf16", n_v=1024, grid=32,
                                                    planted_frac=0.25, distractor_frac=0.25, S=8, Q=16),
                      replace(W.TINY_DECODER, d=8192), replace(W.RIFT_POLICY_SKEW, C=(128, 256, 512, 768, 1024)),
                      knn_m=2)
MAX_DIMS_P = np.array([0.0, 0.03, 0.0, 0.5, 1.0, 0.1, 0.0, 0.9], dtype=np.float32)


def test_longest_tiles_and_widest_embeddings(cuda, riftlib):
    wl = MAX_DIMS
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    sel = P.oracle_select(wl, sc, p_ext=MAX_DIMS_P)
    P.assert_margins(sel, wl)
    assert wl.scene.n_v in sel.budgets  # a whole tile is selected
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    p = torch.tensor(MAX_DIMS_P, device=cuda)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], p=p, prefill=False)
    riftlib.sync_status()
    r = pipe.result(n_kept, T)
    assert P.rel_err_rows(r.token_scores.cpu().numpy(), sel.r64.numpy()) < P.SCORE_RTOL
    assert P.max_abs_rel(r.tile_s_raw.cpu(), sel.s64) < P.SCORE_RTOL
    assert P.max_abs_rel(r.tile_s.cpu(), torch.tensor(sel.s_tilde)) < P.SCORE_RTOL
    assert not P.neighbours_match(r.nbr.cpu().numpy(), sel)
    assert r.kept.cpu().tolist() == sel.kept
    assert r.budgets.cpu().tolist() == sel.budgets
    off = r.sel_off.cpu().tolist()
    got = r.sel.cpu().tolist()
    assert [got[off[j]:off[j + 1]] for j in range(n_kept)] == [list(x) for x in sel.sel]
    H0, cu, pos = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    assert T == H0.shape[0] and r.cu_seqlens.cpu().tolist() == list(cu)
    assert r.positions.cpu().tolist() == list(pos)
    assert torch.equal(r.hidden.cpu(), H0)


def test_query_templates_at_the_widest_embedding(cuda, riftlib):
    """Several caption templates (t = l2norm of the mean of the normalised template embeddings) at
    d = 8192, where the template pass holds two rows of d floats in shared memory."""
    d, vocab, n_tmpl, n_phrase, M = 8192, 300, 3, 5, 4
    sc = W.make_scene(replace(MAX_DIMS.scene, N=1, n_v=4, grid=2, M=M), vocab)
    ids = [[(7 * k + 3 * j + 1) % vocab for j in range(n_phrase)] for k in range(n_tmpl)]
    t_ref = O.query_embedding(sc.embed, ids)
    B_ref = O.background_embeddings(sc.embed, sc.bg_ids)
    i32 = dict(dtype=torch.int32, device=cuda)
    t = torch.empty(d, dtype=torch.float32, device=cuda)
    B = torch.empty(M, d, dtype=torch.float32, device=cuda)
    riftlib.query_prep(sc.embed.to(cuda), vocab, d, torch.tensor(sum(ids, []), **i32), n_tmpl, n_phrase,
                       torch.tensor(sc.bg_ids, **i32), M, t, B)
    riftlib.sync_status()
    assert float((t.cpu().double() - t_ref).abs().max()) < 1e-6
    assert float((B.cpu().double() - B_ref).abs().max()) < 1e-6


def test_empty_batches_are_no_ops(cuda, riftlib):
    """T = 0 rows (prefill, attention) and zero sequences (decode) return OK and write nothing."""
    from paper_2609_29029_gb300 import DeviceModel
    dec = W.TINY_DECODER
    dm = DeviceModel(dec, [W.make_layer(dec, l, "cpu") for l in range(dec.n_layers)], W.make_final_norm(dec, "cpu"),
                     cuda, lm_head=W.make_lm_head(dec, "cpu"))
    i32 = dict(dtype=torch.int32, device=cuda)
    sentinel = torch.full((4, dec.d), 3.0, dtype=torch.bfloat16, device=cuda)
    hidden = sentinel.clone()
    cu = torch.zeros(1, **i32)
    pos = torch.zeros(1, **i32)
    need = riftlib.prefill_workspace_bytes(dm.struct, 0, 0, 16)
    ws = torch.empty(max(need, 256), dtype=torch.uint8, device=cuda)
    riftlib.prefill_layers(dm.struct, hidden, 0, cu, 0, 16, pos, ws, need)
    qkv = torch.zeros(4, 3 * dec.d, dtype=torch.float16, device=cuda)
    out = torch.full((4, dec.d), 5.0, dtype=torch.float16, device=cuda)
    riftlib.attention_varlen(qkv, 0, cu, 0, dec.n_heads, dec.head_dim, out, None, 0)
    kv = torch.zeros(dec.n_layers, 2, 1, dec.d, dtype=torch.float16, device=cuda)
    ids = torch.zeros(1, **i32)
    logits = torch.full((1, dec.vocab), 7.0, dtype=torch.float32, device=cuda)
    embed = W.make_scene(W.TINY.scene, dec.vocab).embed.to(cuda)
    dneed = riftlib.decode_workspace_bytes(dm.struct, 0, 16)
    dws = torch.empty(max(dneed, 256), dtype=torch.uint8, device=cuda)
    riftlib.decode_step(dm.struct, kv, 0, cu, 0, 16, ids, embed, dec.vocab, hidden, None, logits, dws, dneed)
    riftlib.sync_status()
    assert torch.equal(hidden, sentinel)
    assert bool((out == 5.0).all()) and bool((logits == 7.0).all())
