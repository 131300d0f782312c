"""One scene query sharded over R ranks on one GPU: the ranks' protocols (paper_2609_29029_gb300.shard)
run in lockstep in this process, each with its own shard of tiles and the CUDA engine; the
exchanges are served in process (no waiting between kernels: every exchange happens on the host
between launches).  The union over the ranks must equal the single-rank CUDA path bit for bit
(scores of the shard's tiles, neighbours, smoothed scores, u, kept tiles, budgets, selected
tokens, packed rows) and the oracle's selection; the prefilled sequences match the oracle.
"""
import numpy as np
import pytest
import torch

from oracle import rift_oracle as O
from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _single(wl, sc, cuda):
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], prefill=False)
    return pipe.result(n_kept, T), dv


def _sharded(wl, sc, dv, R, cuda, model=None):
    from paper_2609_29029_gb300 import shard
    s = wl.scene
    b = shard.shard_bounds(s.N, R)
    engines = [shard.CudaShardEngine(dv["X"][b[r]:b[r + 1]], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], s.M,
                                     s.S, s.Q, wl.knn_m, wl.policy, model=model) for r in range(R)]
    dec = wl.decoder if model is not None else None
    return shard.run_inprocess([shard.sharded_query(e, r, R, s.N, dec=dec) for r, e in enumerate(engines)])


# sweep6400 over 3 ranks: the whole scene finalises its tiles inside the token pass, the shards of
# 2133 tiles in the separate kernel; both must give the same bits
@pytest.mark.parametrize("name,R", [("small24_f32", 2), ("ragged40_bf16", 3), ("sweep400", 4), ("sweep1600", 3),
                                    ("sweep6400", 3)])
def test_sharded_selection_equals_single_rank(name, R, cuda, riftlib):
    wl = {"small24_f32": P.SMALL24, "ragged40_bf16": P.RAGGED, "sweep400": W.sweep_workload(400),
          "sweep1600": W.sweep_workload(1600), "sweep6400": W.sweep_workload(6400)}[name]
    sc = W.make_scene(wl.scene, wl.decoder.vocab, cuda)
    r1, dv = _single(wl, sc, cuda)
    res = _sharded(wl, sc, dv, R, cuda)
    m = wl.m_eff
    kept = [t for x in res for t in x.kept]
    assert kept == r1.kept.cpu().tolist()
    assert [b for x in res for b in x.budgets] == r1.budgets.cpu().tolist()
    off = r1.sel_off.cpu().tolist()
    s_all = r1.sel.cpu().tolist()
    assert [t for x in res for t in x.sel] == [s_all[off[j]:off[j + 1]] for j in range(len(kept))]
    bits = lambda ts: torch.cat([t.float().cpu() for t in ts]).numpy().view(np.uint32)
    assert np.array_equal(bits([x.tile_s for x in res]), r1.tile_s.cpu().numpy().view(np.uint32))
    assert np.array_equal(bits([x.u for x in res]), r1.u.cpu().numpy().view(np.uint32))
    if m > 0:
        assert torch.equal(torch.cat([x.nbr.cpu() for x in res]), r1.nbr.cpu())
    # every kept tile's packed sequence, wherever it went, is the single-rank one
    cu1 = r1.cu_seqlens.cpu().tolist()
    hid1 = r1.hidden.cpu()
    for x in res:
        for j, t in enumerate(x.seq_tiles):
            k = kept.index(t)
            assert torch.equal(x.rows[x.cu[j]:x.cu[j + 1]].cpu(), hid1[cu1[k]:cu1[k + 1]])
    assert sorted(t for x in res for t in x.seq_tiles) == kept


@pytest.mark.parametrize("name,R", [("small24_f32", 3), ("ragged40_bf16", 2)])
def test_sharded_query_with_prefill_matches_oracle(name, R, cuda, riftlib):
    from paper_2609_29029_gb300 import DeviceModel
    wl = {"small24_f32": P.SMALL24, "ragged40_bf16": P.RAGGED}[name]
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    layers = [W.make_layer(wl.decoder, l) for l in range(wl.decoder.n_layers)]
    gf = W.make_final_norm(wl.decoder)
    dm = DeviceModel(wl.decoder, layers, gf, cuda)
    dv = P.to_dev(sc, cuda)
    res = _sharded(wl, sc, dv, R, cuda, model=dm)
    sel = O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy)
    assert [t for x in res for t in x.kept] == sel.kept
    H0, cu, _ = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    errs = []
    for x in res:
        for j, t in enumerate(x.seq_tiles):
            k = sel.kept.index(t)
            ref = O.prefill_sequence(H0[cu[k]:cu[k + 1]], lambda l: layers[l], gf, wl.decoder)
            errs.append(P.max_abs_rel(x.rows[x.cu[j]:x.cu[j + 1]].cpu(), ref))
    assert len(errs) == len(sel.kept) and max(errs) < P.HIDDEN_TOL, errs
