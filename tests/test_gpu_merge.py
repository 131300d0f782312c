"""The merge of Stage 2 (VisionZip's mechanism: keep the dominant tokens, merge the remainder into
contextual tokens) through the C ABI against the oracle.

Exact: kept tiles, budgets, the dominant token sets (budget less the contextual tokens),
contextual counts and offsets, the targets, every packed row except the contextual ones.  The
contextual rows are bf16 means: each element within one bf16 spacing of the oracle's fp64 mean
(a different group assignment moves a mean by far more).  Every assignment decision of the
oracle clears the float-float rescoring bound (checked first).
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

from oracle import rift_oracle as O
from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _merge_wl(wl):
    return replace(wl, policy=replace(wl.policy, ctx_num=10, ctx_den=64))


def _assignment_margin(X_tile, targets, groups):
    """Smallest relative gap between the chosen target's cosine and the best other target's,
    over the tile's non-target tokens (fp64)."""
    x = X_tile.to(torch.float64)
    xt = x[targets]
    xt = xt / xt.norm(dim=1, keepdim=True)
    worst = np.inf
    for j, gr in enumerate(groups):
        for k in gr[1:]:
            sims = (xt @ x[k]) / x[k].norm()
            others = torch.cat([sims[:j], sims[j + 1:]])
            if len(others):
                worst = min(worst, float(sims[j] - others.max()))
    return worst


def _bf16_close(got, ref):
    """Every element of got (bf16) within one bf16 spacing of the fp64 reference."""
    r = ref.to(torch.float64)
    spacing = torch.clamp(r.abs(), min=1e-30) * 2.0 ** -7
    return bool(((got.to(torch.float64) - r).abs() <= spacing).all())


def _check(wl, cuda, tiles=None, sc=None, sel=None):
    sc = sc if sc is not None else W.make_scene(wl.scene, wl.decoder.vocab)
    sel = sel if sel is not None else P.oracle_select(wl, sc)
    amb = set(P.assert_margins(sel, wl, allow_topb=True))  # rank gaps inside the fp32 bound
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], prefill=False)
    r = pipe.result(n_kept, T)
    assert r.kept.cpu().tolist() == sel.kept
    assert r.budgets.cpu().tolist() == sel.budgets
    off = r.sel_off.cpu().tolist()
    s_all = r.sel.cpu().tolist()
    n_v = wl.scene.n_v
    cto = pipe.ctx_off[:n_kept + 1].cpu().tolist()
    tgt = pipe.ctx_target.cpu().tolist()
    for j, (i, idx, b) in enumerate(zip(sel.kept, sel.sel, sel.budgets)):
        m = O.contextual_count(b, n_v, wl.policy)
        assert cto[j + 1] - cto[j] == m, j
        if j in amb:  # a valid top set; its remaining tokens (and so the merge) may differ
            assert P.topb_is_valid(s_all[off[j]:off[j + 1]], sel.r32[i], len(idx)), j
            continue
        assert s_all[off[j]:off[j + 1]] == idx, j
        assert tgt[cto[j]:cto[j + 1]] == sel.ctx_targets[j], j
    check = [j for j in (range(len(sel.kept)) if tiles is None else tiles) if j not in amb]
    for j in check:
        if not sel.ctx_targets[j]:
            continue
        assert _assignment_margin(sc.X[sel.kept[j]], sel.ctx_targets[j], sel.ctx_groups[j]) > 1e-9, j
        assert _bf16_close(pipe.ctx[cto[j]:cto[j + 1]].cpu(), sel.ctx[j]), j
    # packing: lengths S + budget + Q; the contextual rows are the merge's output rows
    cu = r.cu_seqlens.cpu().tolist()
    S, Q = wl.scene.S, wl.scene.Q
    assert [cu[j + 1] - cu[j] for j in range(n_kept)] == [S + b + Q for b in sel.budgets]
    packed = r.hidden.cpu()
    for j in check:
        i, idx = sel.kept[j], sel.sel[j]
        a = cu[j] + S
        assert torch.equal(packed[a:a + len(idx)], sc.X[i][idx].to(torch.bfloat16)), j
        m = cto[j + 1] - cto[j]
        assert torch.equal(packed[a + len(idx):a + len(idx) + m], pipe.ctx[cto[j]:cto[j + 1]].cpu()), j
        assert torch.equal(packed[cu[j]:cu[j] + S], sc.embed[sc.sys_ids].to(torch.bfloat16))
    return sel, pipe


@pytest.mark.parametrize("wl", [W.TINY, P.SMALL24, P.RAGGED], ids=lambda w: w.name)
def test_merge_matches_oracle(wl, cuda, riftlib):
    _check(_merge_wl(wl), cuda)


def test_merge_at_the_400_tile_scene(cuda, riftlib):
    # every count, target and dominant set; the contextual means of 6 sampled kept tiles
    wl = _merge_wl(P.parity_workload(W.RIFT400))
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    sel = P.oracle_select(wl, sc)
    rnd = np.random.default_rng(0)
    tiles = sorted(rnd.choice(len(sel.kept), size=min(6, len(sel.kept)), replace=False).tolist())
    _check(wl, cuda, tiles=tiles, sc=sc, sel=sel)


def test_merge_off_leaves_selection_and_packing_unchanged(cuda, riftlib):
    wl = P.SMALL24
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    assert pipe.max_m == 0 and pipe.ctx is None
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], prefill=False)
    sel = P.oracle_select(wl, sc)
    H0, cu, _ = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    assert pipe.cu[:n_kept + 1].cpu().tolist() == cu
    assert torch.equal(pipe.packed[:T].cpu(), H0)
