"""The p_i predictor's features (Section 2.3, Stage 2) through the C ABI against the oracle:
quadrant Eq. 1 scores within the score tolerance (1e-4 of the scene's largest), token-score
statistics, and the tile embedding."""
import numpy as np
import pytest
import torch

from oracle import rift_oracle as O
from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _oracle_features(sc, sel, tiles):
    out = []
    for i in tiles:
        q = O.quadrant_scores(sc.X[i], sel.t, sel.B).numpy()
        out.append(np.concatenate([q, np.array(O.token_stats(sel.r32[i]))]))
    return np.array(out)


@pytest.mark.parametrize("wl", [W.TINY, P.SMALL24], ids=lambda w: w.name)
def test_features_of_every_tile_and_of_the_kept_ones(wl, cuda, riftlib):
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    sel = P.oracle_select(wl, sc)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    pipe.select(dv["X"], dv["embed"], dv["q"], dv["bg"])
    V = torch.empty(wl.scene.N, wl.scene.d, dtype=torch.float32, device=cuda)
    f_all = pipe.features(dv["X"], kept_only=False, V=V).cpu().numpy()
    n_kept = int(pipe.n_kept.item())
    f_kept = pipe.features(dv["X"], kept_only=True).cpu().numpy()[:n_kept]
    riftlib.sync_status()
    ref = _oracle_features(sc, sel, range(wl.scene.N))
    scale = np.abs(ref[:, :4]).max()
    assert np.abs(f_all[:, :4] - ref[:, :4]).max() < P.SCORE_RTOL * scale
    assert np.abs(f_all[:, 4:] - ref[:, 4:]).max() < 1e-5 * np.abs(ref[:, 4:]).max()
    assert np.array_equal(f_kept, f_all[sel.kept])            # the kept list selects slots
    assert float((V.cpu().double() - sel.V).abs().max()) < 1e-5


def test_features_at_the_400_tile_scene_for_kept_tiles(cuda, riftlib):
    wl = P.parity_workload(W.RIFT400)
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    pipe.select(dv["X"], dv["embed"], dv["q"], dv["bg"])
    f = pipe.features(dv["X"]).cpu().numpy()
    kept = pipe.kept[:int(pipe.n_kept.item())].cpu().tolist()
    riftlib.sync_status()
    t = O.query_embedding(sc.embed, [sc.query_ids])
    B = O.background_embeddings(sc.embed, sc.bg_ids)
    rnd = np.random.default_rng(1)
    for j in sorted(rnd.choice(len(kept), size=min(8, len(kept)), replace=False).tolist()):
        i = kept[j]
        q = O.quadrant_scores(sc.X[i], t, B).numpy()
        r = O.token_relevance(sc.X[i].to(torch.float64), t, B).numpy()
        ref = np.concatenate([q, np.array(O.token_stats(r))])
        assert np.abs(f[j, :4] - ref[:4]).max() < P.SCORE_RTOL * np.abs(q).max() + 1e-6, j
        assert np.abs(f[j, 4:] - ref[4:]).max() < 1e-4 * np.abs(ref[4:]).max(), j


def test_features_need_an_even_square_grid(cuda, riftlib):
    wl = P.RAGGED  # n_v = 200
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    pipe.select(dv["X"], dv["embed"], dv["q"], dv["bg"])
    with pytest.raises(riftlib.RiftError) as e:
        pipe.features(dv["X"])
    assert e.value.status == riftlib.RIFT_ERR_UNSUPPORTED
