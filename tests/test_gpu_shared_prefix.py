"""Prefill over a shared system prompt through the C ABI: the prompt once, then every sequence's
suffix over its cache, against the oracle's whole-sequence prefill (Tiny, every sequence) and its
prefix + extension (a 7B-shaped batch), at the hidden-state tolerance."""
import pytest
import torch

from oracle import rift_oracle as O
from synth import rng, workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _rel(got, ref):
    ref = ref.to(torch.float64)
    return float((got.to(torch.float64).cpu() - ref).abs().max() / ref.abs().max())


def test_shared_prefix_equals_the_whole_prefill_on_tiny(cuda, riftlib):
    from paper_2609_29029_gb300 import DeviceModel
    wl = W.TINY
    dec = wl.decoder
    sc = W.make_scene(wl.scene, dec.vocab)
    layers = [W.make_layer(dec, l, "cpu") for l in range(dec.n_layers)]
    gf = W.make_final_norm(dec, "cpu")
    dm = DeviceModel(dec, layers, gf, cuda)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, model=dm)
    n, T2 = pipe.run_shared_prefix(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"])
    riftlib.sync_status()
    sel = P.oracle_select(wl, sc)
    H0, cu, _ = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    S = wl.scene.S
    assert T2 == H0.shape[0] - n * S
    cu2 = pipe.cu[:n + 1].cpu().tolist()
    get = lambda l: layers[l]
    pre_ref, pre_cache = O.prefill_with_cache(H0[:S], get, gf, dec)
    assert _rel(pipe.prefix_hidden, pre_ref) < P.HIDDEN_TOL
    for l in range(dec.n_layers):
        assert _rel(pipe.prefix_kv[l, 0], pre_cache[l][0]) < P.HIDDEN_TOL
        assert _rel(pipe.prefix_kv[l, 1], pre_cache[l][1]) < P.HIDDEN_TOL
    worst = 0.0
    for j in range(n):
        full = O.prefill_sequence(H0[cu[j]:cu[j + 1]], get, gf, dec)
        got = pipe.packed[cu2[j]:cu2[j + 1]]
        assert got.shape[0] == full.shape[0] - S
        worst = max(worst, _rel(got, full[S:]))
    assert worst < P.HIDDEN_TOL, worst


def test_shared_prefix_at_the_7b_shape(cuda, riftlib):
    from paper_2609_29029_gb300 import DeviceModel
    dec = W.LLAVA7B
    layers = [W.make_layer(dec, l, cuda) for l in range(dec.n_layers)]
    dm = DeviceModel(dec, layers, W.make_final_norm(dec, cuda), cuda, lm_head=W.make_lm_head(dec, cuda))
    del layers
    torch.cuda.empty_cache()
    S, lens = 35, [50, 140]
    d, n, T = dec.d, len(lens), sum(lens)
    vocab = 4096
    embed = rng.normal_f32(7, rng.stream_id("sp-embed"), vocab * d, cuda).view(vocab, d).to(torch.bfloat16)
    sys_ids = torch.arange(100, 100 + S, dtype=torch.int32, device=cuda)
    rows = rng.normal_f32(8, rng.stream_id("sp-rows"), T * d, cuda).view(T, d).to(torch.bfloat16)
    hidden = rows.clone()
    cu = [0, lens[0], T]
    cu_d = torch.tensor(cu, dtype=torch.int32, device=cuda)
    pos = torch.cat([torch.arange(L, dtype=torch.int32, device=cuda) for L in lens])
    pre_h = torch.empty(S, d, dtype=torch.bfloat16, device=cuda)
    pre_kv = torch.empty(dec.n_layers, 2, S, d, dtype=torch.float16, device=cuda)
    last = torch.empty(n, dec.vocab, dtype=torch.float32, device=cuda)
    max_len = S + max(lens)
    need = riftlib.prefill_shared_prefix_workspace_bytes(dm.struct, T, n, max_len, S)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    riftlib.prefill_shared_prefix(dm.struct, sys_ids, S, embed, vocab, pre_h, pre_kv, hidden, T, cu_d, n, max_len,
                                  pos, last, ws, need)
    riftlib.sync_status()
    # oracle, layer by layer: prefix with its cache, then each suffix over it
    hp = embed[100:100 + S].cpu().to(torch.float64)
    hs = {j: rows[cu[j]:cu[j + 1]].cpu().to(torch.float64) for j in range(n)}
    for l in range(dec.n_layers):
        W64 = {k: v.cpu().to(torch.float64) for k, v in W.make_layer(dec, l, cuda).items()}
        hp, k, v = O.decoder_layer_cached(hp, W64, dec, torch.arange(S))
        for j in range(n):
            hs[j], _, _ = O.decoder_layer_cached(hs[j], W64, dec, torch.arange(S, S + lens[j]), k, v)
        del W64
    gf = W.make_final_norm(dec, cuda).cpu().to(torch.float64)
    lm = W.make_lm_head(dec, cuda).cpu()
    errs = [_rel(pre_h, O.rmsnorm(hp, gf, dec.eps))]
    for j in range(n):
        ref = O.rmsnorm(hs[j], gf, dec.eps)
        errs += [_rel(hidden[cu[j]:cu[j + 1]], ref), _rel(last[j], O.logits(ref[-1], lm))]
    assert max(errs) < P.HIDDEN_TOL, errs
