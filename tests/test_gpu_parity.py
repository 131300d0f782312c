"""Parity of the CUDA path (through the C ABI) with the CPU oracle, at sizes the oracle finishes
in seconds: several tiles, pruning, ragged budgets and tails, both input dtypes.

Integers (kept tiles, neighbours, budgets, token indices, offsets, packed rows) must match
bit-exactly; scores within 1e-4 of the largest magnitude of their row; final hidden states
within 2e-2 max-abs-rel per sequence.
"""
import numpy as np
import pytest
import torch

from oracle import rift_oracle as O
from synth import rng, workloads as W

import parity as P

pytestmark = pytest.mark.gpu

WORKLOADS = [W.TINY, P.SMALL24, P.RAGGED]
HD128 = W.DecoderShape(n_layers=2, d=256, n_heads=2, head_dim=128, ffn=688, vocab=1000)


@pytest.fixture(scope="module")
def cases():
    out = {}
    for wl in WORKLOADS:
        sc = W.make_scene(wl.scene, wl.decoder.vocab)
        sel = P.oracle_select(wl, sc)
        P.assert_margins(sel, wl)
        out[wl.name] = (wl, sc, sel)
    return out


def _model(dec, device):
    from paper_2609_29029_gb300 import DeviceModel
    layers = [W.make_layer(dec, l, "cpu") for l in range(dec.n_layers)]
    gf = W.make_final_norm(dec, "cpu")
    return DeviceModel(dec, layers, gf, device), layers, gf


def test_generator_is_device_independent(cuda):
    spec = W.TINY.scene
    a = W.make_scene(spec, 1000, "cpu")
    b = W.make_scene(spec, 1000, cuda)
    assert torch.equal(a.X, b.X.cpu()) and torch.equal(a.embed, b.embed.cpu())
    wa, wb = W.make_layer(W.TINY_DECODER, 1, "cpu"), W.make_layer(W.TINY_DECODER, 1, cuda)
    assert all(torch.equal(wa[k], wb[k].cpu()) for k in wa)


@pytest.mark.parametrize("name", [w.name for w in WORKLOADS])
def test_scores_and_selection_match_oracle(name, cases, cuda, riftlib):
    wl, sc, sel = cases[name]
    pipe, dv = P.gpu_pipeline(wl, sc, cuda)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], prefill=False)
    r = pipe.result(n_kept, T)
    # a1: query embedding
    assert float((r.t.cpu().double() - sel.t).abs().max()) < 1e-6
    # a2, a3: scores within tolerance
    assert P.rel_err_rows(r.token_scores.cpu().numpy(), sel.r64.numpy()) < P.SCORE_RTOL
    assert P.max_abs_rel(r.tile_s_raw.cpu(), sel.s64) < P.SCORE_RTOL
    assert P.max_abs_rel(r.tile_s.cpu(), torch.tensor(sel.s_tilde)) < P.SCORE_RTOL
    # a4-a7: every decision exact
    if wl.m_eff > 0:
        assert not P.neighbours_match(r.nbr.cpu().numpy(), sel)
    assert n_kept == len(sel.kept)
    assert r.kept.cpu().tolist() == sel.kept
    assert r.budgets.cpu().tolist() == sel.budgets
    off = r.sel_off.cpu().tolist()
    assert off == [0] + list(np.cumsum(sel.budgets))
    s_all = r.sel.cpu().tolist()
    for j, idx in enumerate(sel.sel):
        assert s_all[off[j]:off[j + 1]] == idx
    # a8: packing, bit-exact
    H0, cu, pos = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    assert T == H0.shape[0] and r.cu_seqlens.cpu().tolist() == cu
    assert r.positions.cpu().tolist() == pos
    assert torch.equal(r.hidden.cpu(), H0)


def _select_inputs(N, n_v, seed, ties=True):
    key = rng.stream_id("select-test", seed)
    r = rng.uniform_f32(seed, key, N * n_v).view(N, n_v)
    s = rng.uniform_f32(seed, key + 1, N)
    if ties:  # coarse values force equal keys; add signed zeros
        r = torch.floor(r * 16) / 16 - 0.5
        r.view(-1)[::37] = -0.0
        r.view(-1)[::41] = 0.0
        s = torch.floor(s * 8) / 8
    return r.contiguous(), s.contiguous()


def _run_select(riftlib, r, s, policy, p, cuda):
    N, n_v = r.shape
    dev = dict(device=cuda)
    u = torch.empty(N, dtype=torch.float32, **dev)
    kept = torch.empty(N, dtype=torch.int32, **dev)
    n_kept = torch.empty(1, dtype=torch.int32, **dev)
    bud = torch.empty(N, dtype=torch.int32, **dev)
    sel = torch.full((N * n_v,), -1, dtype=torch.int32, **dev)
    off = torch.empty(N + 1, dtype=torch.int32, **dev)
    rd, sd = r.to(cuda), s.to(cuda)
    pd = p.to(cuda) if p is not None else None
    riftlib.select_budgeted_tokens(rd, sd, N, n_v, pd, riftlib.make_policy(policy), u, kept, n_kept, bud, sel, off,
                                   None, 0)
    riftlib.sync_status()
    n = int(n_kept.item())
    return u.cpu().numpy(), kept[:n].cpu().tolist(), bud[:n].cpu().tolist(), sel.cpu().tolist(), off.cpu().tolist()


def _oracle_select_only(r, s, policy, p):
    r32, s32 = r.numpy().astype(np.float32), s.numpy().astype(np.float32)
    u = O.minmax_normalize(s32)
    kept = O.retained(u, policy.tau)
    pv = [u[i] if p is None else np.float32(p[i]) for i in kept]
    bud = [O.budget(float(x), policy) for x in pv]
    sel = [O.top_b(r32[i], b) for i, b in zip(kept, bud)]
    return u, kept, bud, sel


SELECT_CASES = [
    ("ties", 50, 576, W.RIFT_POLICY, False, True),
    ("single_tile", 1, 576, W.RIFT_POLICY, False, True),
    ("keep_all_full", 30, 576, W.KEEP_ALL, False, True),
    ("tau_one", 64, 576, W.Policy(1.0, (16, 100), (0.9, 0.8), (0.5, 0.9), (0.1, 1.0), 0.1), False, True),
    ("ragged_nv", 33, 1000, W.RIFT_POLICY_SKEW, False, False),
    ("ext_p", 77, 576, W.RIFT_POLICY_SKEW, True, True),
    ("many_tiles", 3000, 64, W.Policy(0.2, (1, 8, 16, 64), (0.9, 0.9, 0.9, 0.9), (0.2, 0.5, 0.7, 0.9),
                                        (0.1, 0.2, 0.4, 1.0), 0.2), False, True),
]


@pytest.mark.parametrize("case", SELECT_CASES, ids=[c[0] for c in SELECT_CASES])
def test_selection_is_bit_exact_on_shared_fp32_inputs(case, cuda, riftlib):
    name, N, n_v, policy, ext_p, ties = case
    r, s = _select_inputs(N, n_v, 7, ties)
    if name == "single_tile":
        s = s[:1]
    p = rng.uniform_f32(3, 99, N) if ext_p else None
    gu, gk, gb, gs, goff = _run_select(riftlib, r, s, policy, p, cuda)
    ou, ok, ob, osel = _oracle_select_only(r, s, policy, p)
    assert np.array_equal(gu.view(np.uint32), ou.view(np.uint32))
    assert gk == ok and gb == ob
    assert goff[:len(ok) + 1] == [0] + list(np.cumsum(ob)) and all(v == sum(ob) for v in goff[len(ok):])
    for j, idx in enumerate(osel):
        assert gs[goff[j]:goff[j + 1]] == idx


def test_selection_all_scores_equal(cuda, riftlib):
    r = torch.zeros(10, 576)
    s = torch.full((10,), 0.25)
    gu, gk, gb, gs, goff = _run_select(riftlib, r, s, W.RIFT_POLICY, None, cuda)
    assert np.all(gu == 1.0) and gk == list(range(10)) and gb == [72] * 10
    assert gs[:72] == list(range(72))


def test_nonfinite_score_is_reported(cuda, riftlib):
    r, s = _select_inputs(8, 576, 1)
    s[3] = float("nan")
    with pytest.raises(riftlib.RiftError) as e:
        _run_select(riftlib, r, s, W.RIFT_POLICY, None, cuda)
    assert e.value.status == riftlib.RIFT_ERR_NONFINITE
    riftlib.sync_status()  # the flag was cleared


@pytest.mark.parametrize("name", [w.name for w in WORKLOADS])
def test_pack_capacity_is_enforced(name, cases, cuda, riftlib):
    wl, sc, sel = cases[name]
    T = sum(wl.scene.S + b + wl.scene.Q for b in sel.budgets)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, max_T=T - 1)
    pipe.select(dv["X"], dv["embed"], dv["q"], dv["bg"])
    pipe.pack(dv["X"], dv["embed"], dv["sys"], dv["q"])
    with pytest.raises(riftlib.RiftError) as e:
        riftlib.sync_status()
    assert e.value.status == riftlib.RIFT_ERR_CAPACITY


def _prefill_gpu(riftlib, dm, H0, cu, pos, max_len, cuda):
    T = H0.shape[0]
    hid = H0.to(cuda).contiguous()
    cu_d = torch.tensor(cu, dtype=torch.int32, device=cuda)
    pos_d = torch.tensor(pos, dtype=torch.int32, device=cuda)
    need = riftlib.prefill_workspace_bytes(dm.struct, T, len(cu) - 1, max_len)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    riftlib.prefill_layers(dm.struct, hid, T, cu_d, len(cu) - 1, max_len, pos_d, ws, need)
    riftlib.sync_status()
    return hid.cpu()


@pytest.mark.parametrize("dec", [W.TINY_DECODER, HD128], ids=["hd64", "hd128"])
def test_prefill_matches_oracle_on_awkward_lengths(dec, cuda, riftlib):
    lengths = [1, 2, 63, 64, 65, 130, 200]
    T = sum(lengths)
    H0 = (rng.normal_f32(0, rng.stream_id("h0"), T * dec.d).view(T, dec.d)).to(torch.bfloat16)
    cu = [0] + list(np.cumsum(lengths))
    pos = [p for L in lengths for p in range(L)]
    dm, layers, gf = _model(dec, cuda)
    out = _prefill_gpu(riftlib, dm, H0, cu, pos, max(lengths), cuda)
    for a, b in P.seq_slices(cu):
        ref = O.prefill_sequence(H0[a:b], lambda l: layers[l], gf, dec)
        assert P.max_abs_rel(out[a:b], ref) < P.HIDDEN_TOL, (a, b)


@pytest.mark.parametrize("name", [w.name for w in WORKLOADS])
def test_end_to_end_matches_oracle(name, cases, cuda, riftlib):
    wl, sc, sel = cases[name]
    dm, layers, gf = _model(wl.decoder, cuda)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, model=dm)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"])
    r = pipe.result(n_kept, T)
    assert r.kept.cpu().tolist() == sel.kept and r.budgets.cpu().tolist() == sel.budgets
    H0, cu, pos = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    out = r.hidden.cpu()
    errs = []
    for a, b in P.seq_slices(cu):
        ref = O.prefill_sequence(H0[a:b], lambda l: layers[l], gf, wl.decoder)
        errs.append(P.max_abs_rel(out[a:b], ref))
    assert max(errs) < P.HIDDEN_TOL, errs


def test_full_budget_equals_exhaustive_prefill_bit_for_bit(cases, cuda, riftlib):
    # tau = 0 and C = {n_v} through the whole Rift path must give exactly the exhaustive
    # tiled prefill: every tile packed as [system | all tokens | query], no token dropped.
    wl, sc, _ = cases[P.SMALL24.name]
    wl = P.with_policy(wl, W.KEEP_ALL)
    dm, layers, gf = _model(wl.decoder, cuda)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, model=dm)
    n_kept, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"])
    rift_out = pipe.result(n_kept, T).hidden.cpu().clone()
    N, S, Q = wl.scene.N, wl.scene.S, wl.scene.Q
    exh = torch.cat([torch.cat([sc.embed[sc.sys_ids], sc.X[i].to(torch.bfloat16), sc.embed[sc.query_ids]])
                     for i in range(N)])
    L = S + 576 + Q
    cu = [L * i for i in range(N + 1)]
    pos = list(range(L)) * N
    exh_out = _prefill_gpu(riftlib, dm, exh, cu, pos, L, cuda)
    assert n_kept == N and T == exh.shape[0]
    assert torch.equal(rift_out, exh_out)


@pytest.mark.parametrize("name", [P.SMALL24.name, P.RAGGED.name])
def test_device_counts_equal_host_counts(name, cases, cuda, riftlib):
    """The query enqueued whole, the prefill reading n_kept and T on the device (no host
    read-back), gives the same final hidden states bit for bit as the prefill run with the counts
    read back to the host.  Both batches have more than 1024 rows, so both take the same GEMM
    path (SM pairs)."""
    wl, sc, sel = cases[name]
    dm, layers, gf = _model(wl.decoder, cuda)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, model=dm)
    args = (dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"])
    assert pipe.run(*args, counts=False) is None
    n_kept, T = pipe.counts()
    riftlib.sync_status()
    assert T >= 1024 and T == sum(wl.scene.S + b + wl.scene.Q for b in sel.budgets)
    dev_out = pipe.packed[:T].cpu().clone()
    pipe.run(*args, prefill=False)
    pipe.prefill(counts=(n_kept, T))
    riftlib.sync_status()
    assert torch.equal(pipe.packed[:T].cpu(), dev_out)


def test_device_sequence_count_above_capacity_is_reported(cuda, riftlib):
    """A device sequence count above max_seqs: the first max_seqs sequences are prefilled and
    the next rift_sync_status returns RIFT_ERR_CAPACITY; the context stays usable."""
    dec = W.TINY_DECODER
    dm, layers, gf = _model(dec, cuda)
    lengths = [40, 24]
    T = sum(lengths)
    H0 = rng.normal_f32(11, rng.stream_id("count-cap"), T * dec.d, "cpu").view(T, dec.d).to(torch.bfloat16)
    cu = torch.tensor([0, 40, 64], dtype=torch.int32, device=cuda)
    pos = torch.tensor(list(range(40)) + list(range(24)), dtype=torch.int32, device=cuda)
    i32 = dict(dtype=torch.int32, device=cuda)
    need = riftlib.prefill_workspace_bytes(dm.struct, T, 1, 64)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    hid = H0.to(cuda)
    riftlib.prefill_layers(dm.struct, hid, torch.tensor([T], **i32), cu, torch.tensor([2], **i32), 64, pos, ws,
                           need, max_T=T, max_seqs=1)
    with pytest.raises(riftlib.RiftError) as e:
        riftlib.sync_status()
    assert e.value.status == riftlib.RIFT_ERR_CAPACITY
    ref = O.prefill_sequence(H0[:40], lambda l: layers[l], gf, dec)
    assert P.max_abs_rel(hid[:40].cpu(), ref) < P.HIDDEN_TOL
    riftlib.sync_status()  # cleared
