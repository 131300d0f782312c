"""Degenerate scenes through the whole CUDA path against the oracle: one tile (min-max has no
spread, so u = 1 and the tile is kept; no neighbours), two tiles without background terms (Eq. 1
is the plain cosine; smoothing over the one neighbour makes both scores equal, so u = 1 for
both), no smoothing (m = 0), and nine tiles with one planted."""
from dataclasses import replace

import pytest

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
