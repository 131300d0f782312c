"""Several scene queries in one prefill: each query packed after the rows of the ones before it
(rift_pack_ragged_at) and the whole batch prefilled at once.  The queries' sequences are
independent (no attention across them), so each query's selection, offsets and final hidden
states must be those of the query run alone, and match the oracle."""
from dataclasses import replace

import pytest
import torch

from oracle import rift_oracle as O
from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu

# three different scenes and queries (seeds) of each workload; the tiny queries alone stay under
# 1024 rows (products on single SMs) while their batch passes it (products on SM pairs)
SEEDS = (0, 1, 2)


def _model(dec, device):
    from paper_2609_29029_gb300 import DeviceModel
    layers = [W.make_layer(dec, l, "cpu") for l in range(dec.n_layers)]
    gf = W.make_final_norm(dec, "cpu")
    return DeviceModel(dec, layers, gf, device), layers, gf


def _query(sc, dv):
    return (dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"])


@pytest.mark.parametrize("base", [P.SMALL24, W.TINY], ids=["small24", "tiny"])
def test_batched_queries_match_their_single_runs_and_the_oracle(base, cuda, riftlib):
    dm, layers, gf = _model(base.decoder, cuda)
    wls = [replace(base, scene=replace(base.scene, seed=s)) for s in SEEDS]
    scenes = [W.make_scene(wl.scene, wl.decoder.vocab) for wl in wls]
    pipe, _ = P.gpu_pipeline(wls[0], scenes[0], cuda, model=dm)
    devs = [P.to_dev(sc, cuda) for sc in scenes]
    res = pipe.run_batch([_query(sc, dv) for sc, dv in zip(scenes, devs)])
    riftlib.sync_status()
    rows = res[-1][1] + res[-1][2]
    seqs = res[-1][0] + res[-1][3]
    batch_hidden = pipe.batch_packed[:rows].cpu().clone()
    batch_cu = pipe.batch_cu[:seqs + 1].cpu().tolist()
    batch_pos = pipe.batch_positions[:rows].cpu().tolist()

    for (wl, sc, dv), (n_kept, T, row0, seq0) in zip(zip(wls, scenes, devs), res):
        # the query alone
        single, _ = P.gpu_pipeline(wl, sc, cuda, model=dm)
        n1, T1 = single.run(*_query(sc, dv))
        r = single.result(n1, T1)
        assert (n_kept, T) == (n1, T1)
        assert batch_cu[seq0:seq0 + n_kept + 1] == [row0 + v for v in r.cu_seqlens.cpu().tolist()]
        assert batch_pos[row0:row0 + T] == r.positions.cpu().tolist()
        mine = batch_hidden[row0:row0 + T]
        alone = r.hidden.cpu()
        assert P.max_abs_rel(mine, alone.float()) < 1e-3
        # and the oracle
        sel = O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy)
        assert r.kept.cpu().tolist() == sel.kept and r.budgets.cpu().tolist() == sel.budgets
        H0, cu, _ = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
        errs = [P.max_abs_rel(mine[a:b], O.prefill_sequence(H0[a:b], lambda l: layers[l], gf, wl.decoder))
                for a, b in P.seq_slices(cu)]
        assert max(errs) < P.HIDDEN_TOL, errs
    assert batch_cu[seqs] == rows

