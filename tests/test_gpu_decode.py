"""The prefill's optional outputs (KV cache, last-token logits) and the decode step, through the
C ABI, against the oracle (Section 2.1): every sequence of the Tiny workload, both head sizes.

Tolerance: the same 2e-2 max-abs-rel per sequence as the final hidden states (the cache and the
logits are fp16 / fp32 results of the same fp16-operand path); decode outputs likewise, with the
GPU decoding from its own fp16 cache and the oracle from its fp64 cache.
"""
import pytest
import torch

from oracle import rift_oracle as O
from synth import rng, workloads as W

import parity as P

pytestmark = pytest.mark.gpu

HD128 = W.DecoderShape(n_layers=2, d=256, n_heads=2, head_dim=128, ffn=688, vocab=1000)


def _model(dec, device):
    from paper_2609_29029_gb300 import DeviceModel
    layers = [W.make_layer(dec, l, "cpu") for l in range(dec.n_layers)]
    gf = W.make_final_norm(dec, "cpu")
    lm = W.make_lm_head(dec, "cpu")
    return DeviceModel(dec, layers, gf, device, lm_head=lm), layers, gf, lm


def _rel(got, ref):
    ref = ref.to(torch.float64)
    return float((got.to(torch.float64).cpu() - ref).abs().max() / ref.abs().max())


def _token_ids(n, vocab, seed):
    key = rng.stream_key(seed, rng.stream_id("decode-ids"))
    return [rng.hash_u32_int(key, i) % vocab for i in range(n)]


@pytest.mark.parametrize("dec", [W.TINY_DECODER, HD128], ids=["hd64", "hd128"])
def test_cache_logits_and_decode_match_oracle(dec, cuda, riftlib):
    wl = W.TINY
    sc = W.make_scene(wl.scene, dec.vocab)
    dm, layers, gf, lm = _model(dec, cuda)
    pipe, dv = P.gpu_pipeline(wl, sc, cuda, model=dm)
    n, T = pipe.run(dv["X"], dv["embed"], dv["q"], dv["bg"], dv["sys"], dv["q"], prefill=False)
    packed = pipe.packed[:T].cpu().clone()
    kv = torch.full((dec.n_layers, 2, T, dec.d), float("nan"), dtype=torch.float16, device=cuda)
    last = torch.full((n, dec.vocab), float("nan"), dtype=torch.float32, device=cuda)
    pipe.prefill(kv_out=kv, last_logits=last, counts=(n, T))
    ids = _token_ids(n, dec.vocab, 1)
    ids_d = torch.tensor(ids, dtype=torch.int32, device=cuda)
    hid = torch.empty(n, dec.d, dtype=torch.bfloat16, device=cuda)
    kvn = torch.empty(dec.n_layers, 2, n, dec.d, dtype=torch.float16, device=cuda)
    lg = torch.empty(n, dec.vocab, dtype=torch.float32, device=cuda)
    pipe.decode(kv, T, n, ids_d, dv["embed"], hid, kvn, lg)
    riftlib.sync_status()
    cu = pipe.cu[:n + 1].cpu().tolist()
    get = lambda l: layers[l]
    worst = {}
    for j in range(n):
        h_ref, cache = O.prefill_with_cache(packed[cu[j]:cu[j + 1]], get, gf, dec)
        errs = [_rel(pipe.packed[cu[j]:cu[j + 1]], h_ref), _rel(last[j], O.logits(h_ref[-1], lm))]
        for l in range(dec.n_layers):
            errs += [_rel(kv[l, 0, cu[j]:cu[j + 1]], cache[l][0]), _rel(kv[l, 1, cu[j]:cu[j + 1]], cache[l][1])]
        hd, new = O.decode_token(sc.embed[ids[j]], cache, get, gf, dec)
        errs += [_rel(hid[j], hd), _rel(lg[j], O.logits(hd, lm))]
        for l in range(dec.n_layers):
            errs += [_rel(kvn[l, 0, j], new[l][0]), _rel(kvn[l, 1, j], new[l][1])]
        worst[j] = max(errs)
    assert max(worst.values()) < P.HIDDEN_TOL, worst


def test_decode_with_an_empty_prompt_is_a_one_token_prefill(cuda, riftlib):
    # L_i = 0: the token attends to itself only, at position 0.
    dec = W.TINY_DECODER
    dm, layers, gf, lm = _model(dec, cuda)
    embed = (rng.normal_f32(3, rng.stream_id("dec-embed"), 50 * dec.d, cuda).view(50, dec.d)).to(torch.bfloat16)
    cu = torch.zeros(3, dtype=torch.int32, device=cuda)
    ids = torch.tensor([7, 41], dtype=torch.int32, device=cuda)
    kv = torch.zeros(8, dtype=torch.float16, device=cuda)  # never read: no cached rows
    hid = torch.empty(2, dec.d, dtype=torch.bfloat16, device=cuda)
    lg = torch.empty(2, dec.vocab, dtype=torch.float32, device=cuda)
    need = riftlib.decode_workspace_bytes(dm.struct, 2, 4)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    riftlib.decode_step(dm.struct, kv, 0, cu, 2, 4, ids, embed, 50, hid, None, lg, ws, need)
    riftlib.sync_status()
    for j, t in enumerate((7, 41)):
        ref = O.prefill_sequence(embed[t:t + 1].cpu(), lambda l: layers[l], gf, dec)[0]
        assert _rel(hid[j], ref) < P.HIDDEN_TOL
        assert _rel(lg[j], O.logits(ref, lm)) < P.HIDDEN_TOL


def test_decode_flags_bad_ids_and_short_max_len(cuda, riftlib):
    dec = W.TINY_DECODER
    dm, _, _, _ = _model(dec, cuda)
    T = 10
    cu = torch.tensor([0, 4, 10], dtype=torch.int32, device=cuda)
    kv = torch.zeros(dec.n_layers, 2, T, dec.d, dtype=torch.float16, device=cuda)
    embed = torch.zeros(20, dec.d, dtype=torch.bfloat16, device=cuda)
    hid = torch.empty(2, dec.d, dtype=torch.bfloat16, device=cuda)

    def run(ids, max_len):
        need = riftlib.decode_workspace_bytes(dm.struct, 2, max_len)
        ws = torch.empty(need, dtype=torch.uint8, device=cuda)
        riftlib.decode_step(dm.struct, kv, T, cu, 2, max_len, torch.tensor(ids, dtype=torch.int32, device=cuda),
                            embed, 20, hid, None, None, ws, need)
        return riftlib.lib.rift_sync_status(None)

    assert run([3, 5], 11) == riftlib.RIFT_OK
    assert run([3, 20], 11) == riftlib.RIFT_ERR_BAD_ID          # id == vocab_embed
    assert run([-1, 5], 11) == riftlib.RIFT_ERR_BAD_ID
    assert run([3, 5], 7) == riftlib.RIFT_OK                    # L = 6 at position 6, 7 keys
    assert run([3, 5], 6) in (riftlib.RIFT_ERR_BAD_ID, riftlib.RIFT_ERR_CAPACITY)   # position 6 >= max_len
    assert run([3, 5], 11) == riftlib.RIFT_OK                   # flags were cleared
    # host-checked arguments
    need = riftlib.decode_workspace_bytes(dm.struct, 2, 11)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    ids = torch.tensor([3, 5], dtype=torch.int32, device=cuda)
    st = riftlib.lib.rift_decode_step(riftlib.C.byref(dm.struct), kv.data_ptr(), T, cu.data_ptr(), 2, 11,
                                      ids.data_ptr(), embed.data_ptr(), 20, None, None, 1, ws.data_ptr(), need, None)
    assert st == riftlib.RIFT_ERR_INVALID                        # misaligned logits pointer


# d = 1024 with 4 heads of 128 and one layer: every GEMM of the decode step (a few rows) runs
# split-K (QKV with RoPE 4 slices, W_o 4, gate/up with SwiGLU 4, W_down 11, output matrix 4),
# the prefill's GEMMs do not.
MID = W.DecoderShape(n_layers=1, d=1024, n_heads=8, head_dim=128, ffn=2816, vocab=4096)


def test_split_k_decode_on_a_synthetic_batch(cuda, riftlib):
    dec = MID
    dm, layers, gf, lm = _model(dec, cuda)
    lens = [5, 64, 130]
    T, n, d = sum(lens), len(lens), dec.d
    cu = [0, 5, 69, T]
    H0 = rng.normal_f32(11, rng.stream_id("mid-batch"), T * d, cuda).view(T, d).to(torch.bfloat16)
    hidden = H0.clone()
    cu_d = torch.tensor(cu, dtype=torch.int32, device=cuda)
    pos_d = torch.cat([torch.arange(L, dtype=torch.int32, device=cuda) for L in lens])
    kv = torch.empty(dec.n_layers, 2, T, d, dtype=torch.float16, device=cuda)
    last = torch.empty(n, dec.vocab, dtype=torch.float32, device=cuda)
    max_len = max(lens) + 1
    need = riftlib.prefill_workspace_bytes(dm.struct, T, n, max_len)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    riftlib.prefill_layers(dm.struct, hidden, T, cu_d, n, max_len, pos_d, ws, need, kv_out=kv, last_logits=last)
    embed = rng.normal_f32(12, rng.stream_id("mid-embed"), 300 * d, cuda).view(300, d).to(torch.bfloat16)
    ids = _token_ids(n, 300, 2)
    hid = torch.empty(n, d, dtype=torch.bfloat16, device=cuda)
    kvn = torch.empty(dec.n_layers, 2, n, d, dtype=torch.float16, device=cuda)
    lg = torch.empty(n, dec.vocab, dtype=torch.float32, device=cuda)
    need = riftlib.decode_workspace_bytes(dm.struct, n, max_len)
    ws = torch.empty(need, dtype=torch.uint8, device=cuda)
    riftlib.decode_step(dm.struct, kv, T, cu_d, n, max_len, torch.tensor(ids, dtype=torch.int32, device=cuda),
                        embed, 300, hid, kvn, lg, ws, need)
    riftlib.sync_status()
    # the reductions inside the products and the attention leave their arrival counters zeroed:
    # a second step on the same workspace gives the same bits
    hid2, kvn2, lg2 = torch.empty_like(hid), torch.empty_like(kvn), torch.empty_like(lg)
    riftlib.decode_step(dm.struct, kv, T, cu_d, n, max_len, torch.tensor(ids, dtype=torch.int32, device=cuda),
                        embed, 300, hid2, kvn2, lg2, ws, need)
    riftlib.sync_status()
    assert torch.equal(hid, hid2) and torch.equal(kvn, kvn2) and torch.equal(lg, lg2)
    get = lambda l: layers[l]
    worst = {}
    for j in range(n):
        h_ref, cache = O.prefill_with_cache(H0[cu[j]:cu[j + 1]].cpu(), get, gf, dec)
        hd, new = O.decode_token(embed[ids[j]].cpu(), cache, get, gf, dec)
        errs = [_rel(hidden[cu[j]:cu[j + 1]], h_ref), _rel(last[j], O.logits(h_ref[-1], lm)),
                _rel(hid[j], hd), _rel(lg[j], O.logits(hd, lm))]
        for l in range(dec.n_layers):
            errs += [_rel(kv[l, 0, cu[j]:cu[j + 1]], cache[l][0]), _rel(kv[l, 1, cu[j]:cu[j + 1]], cache[l][1]),
                     _rel(kvn[l, 0, j], new[l][0]), _rel(kvn[l, 1, j], new[l][1])]
        worst[j] = max(errs)
    print("worst", worst)
    assert max(worst.values()) < P.HIDDEN_TOL, worst
