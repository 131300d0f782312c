"""Pins of the CPU oracle against what the paper and the mathematics fix, not against itself.

Each test names the passage it pins.  None of these needs a GPU.
"""
import itertools
import math
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as F
from scipy.spatial import distance

from oracle import rift_oracle as O
from synth import workloads as W

F32 = np.float32


# ---------------------------------------------------------------- Eq. 1 (Section 2.3 Stage 1)

def test_eq1_hand_case():
    # V = (1, 0), t = (0.6, 0.8), B = {(1, 0), (0, 1)}: s = 0.6 - (1 + 0)/2 = 0.1
    V = torch.tensor([[1.0, 0.0]], dtype=torch.float64)
    t = torch.tensor([0.6, 0.8], dtype=torch.float64)
    B = torch.tensor([[1.0, 0.0], [0.0, 1.0]], dtype=torch.float64)
    assert float(O.margin(V, t, B)[0]) == pytest.approx(0.1, abs=1e-15)


def test_eq1_tile_equal_to_query():
    # V = t gives s = 1 - mean_j B_j . t
    g = torch.Generator().manual_seed(1)
    t = O.l2norm(torch.randn(16, generator=g, dtype=torch.float64))
    B = O.l2norm(torch.randn(5, 16, generator=g, dtype=torch.float64))
    s = O.margin(t[None, :], t, B)
    assert float(s[0]) == pytest.approx(1.0 - float((B @ t).mean()), abs=1e-14)


def test_eq1_without_background_is_cosine():
    # M = 0: s_i = cos(V_i, t) (scipy's cosine distance is 1 - cos)
    rng = np.random.default_rng(2)
    X = rng.standard_normal((7, 33))
    t = rng.standard_normal(33)
    s = O.margin(O.l2norm(torch.tensor(X)), O.l2norm(torch.tensor(t)), torch.zeros(0, 33, dtype=torch.float64))
    ref = [1.0 - distance.cosine(x, t) for x in X]
    np.testing.assert_allclose(s.numpy(), ref, rtol=0, atol=1e-13)


def test_token_relevance_matches_scipy_cosines():
    rng = np.random.default_rng(3)
    X = rng.standard_normal((11, 24))
    t = rng.standard_normal(24)
    B = rng.standard_normal((4, 24))
    r = O.token_relevance(torch.tensor(X), O.l2norm(torch.tensor(t)), O.l2norm(torch.tensor(B)))
    ref = [(1 - distance.cosine(x, t)) - np.mean([1 - distance.cosine(x, b) for b in B]) for x in X]
    np.testing.assert_allclose(r.numpy(), ref, rtol=0, atol=1e-13)


def test_tile_embedding_is_direction_of_the_pooled_tokens():
    rng = np.random.default_rng(4)
    X = torch.tensor(rng.standard_normal((9, 12)))
    V = O.tile_embedding(X)
    s = X.sum(0)
    np.testing.assert_allclose(V.numpy(), (s / s.norm()).numpy(), atol=1e-15)
    np.testing.assert_allclose(O.tile_embedding(3.5 * X).numpy(), V.numpy(), atol=1e-15)
    assert float(V.norm()) == pytest.approx(1.0, abs=1e-15)


def test_query_embedding_templates():
    E = torch.tensor([[3.0, 4.0, 0.0], [0.0, 0.0, 2.0], [1.0, 0.0, 0.0]], dtype=torch.float64)
    # one template, one id: t = E[id] / ||E[id]||
    np.testing.assert_allclose(O.query_embedding(E, [0]).numpy(), [0.6, 0.8, 0.0], atol=1e-15)
    # two templates [0] and [1]: l2norm((0.6, 0.8, 0) + (0, 0, 1)) = (0.6, 0.8, 1)/sqrt(2)
    np.testing.assert_allclose(O.query_embedding(E, [[0], [1]]).numpy(),
                               np.array([0.6, 0.8, 1.0]) / math.sqrt(2), atol=1e-15)
    # one template [0, 2]: mean (2, 2, 0) -> (1, 1, 0)/sqrt(2)
    np.testing.assert_allclose(O.query_embedding(E, [0, 2]).numpy(), np.array([1, 1, 0]) / math.sqrt(2), atol=1e-15)
    B = O.background_embeddings(E, [1, 0])
    np.testing.assert_allclose(B.numpy(), [[0, 0, 1], [0.6, 0.8, 0]], atol=1e-15)


# ---------------------------------------------------------------- kNN smoothing (Appendix B Step 2)

def _beats(G, i, a, b):
    """a ranks before b as a neighbour of i: larger similarity, then the lower index."""
    return G[i, a] > G[i, b] or (G[i, a] == G[i, b] and a < b)


@pytest.mark.parametrize("seed", range(6))
def test_knn_neighbours_brute_force(seed):
    rng = np.random.default_rng(seed)
    N = 7
    G = rng.integers(-3, 4, size=(N, N)).astype(F32)  # small integers force many ties
    for m in range(0, N):
        nbr = O.knn_neighbours(G, m)
        for i in range(N):
            others = [j for j in range(N) if j != i]
            # the unique m-subset whose every member beats every non-member
            sets = [set(S) for S in itertools.combinations(others, m)
                    if all(_beats(G, i, a, b) for a in S for b in others if b not in S)]
            assert len(sets) == 1
            assert set(nbr[i].tolist()) == sets[0]
            # rank order
            assert all(_beats(G, i, nbr[i][k], nbr[i][k + 1]) for k in range(m - 1))


def test_knn_m_capped_at_n_minus_one():
    G = np.eye(3, dtype=F32)
    assert O.knn_neighbours(G, 6).shape == (3, 2)


def test_smooth_hand_case_and_special_cases():
    s = np.array([0.0, 1.0, 2.0, 3.0], dtype=F32)
    nbr = np.array([[1], [0], [3], [2]])
    np.testing.assert_array_equal(O.smooth(s, nbr), np.array([0.5, 0.5, 2.5, 2.5], dtype=F32))
    # m = 0: no smoothing, bit-exact
    np.testing.assert_array_equal(O.smooth(s, np.zeros((4, 0), dtype=np.int64)), s)
    # m = N - 1: every tile averages the whole scene; sums run in index order, so the results
    # are bit-equal and min-max gives u = 1 everywhere
    rng = np.random.default_rng(0)
    s = rng.standard_normal(5).astype(F32)
    nbr = np.array([[j for j in range(5) if j != i] for i in range(5)])[:, ::-1].copy()
    st = O.smooth(s, nbr)
    assert len(set(st.tolist())) == 1
    assert np.all(O.minmax_normalize(st) == 1.0)


# ---------------------------------------------------------------- min-max and tau (Stage 1; App. B Step 3)

def test_minmax_invariants_and_top_tile_kept():
    rng = np.random.default_rng(5)
    for _ in range(20):
        s = rng.standard_normal(rng.integers(2, 50)).astype(F32)
        u = O.minmax_normalize(s)
        assert u.dtype == F32
        assert u[np.argmax(s)] == 1.0 and u[np.argmin(s)] == 0.0
        assert np.all((u >= 0) & (u <= 1))
        kept = O.retained(u, 0.37)
        assert int(np.argmax(s)) in kept  # "no query can be left with zero tiles"


def test_minmax_two_tiles_and_all_equal():
    assert O.minmax_normalize(np.array([0.3, -0.2], dtype=F32)).tolist() == [1.0, 0.0]
    assert O.minmax_normalize(np.array([0.25] * 4, dtype=F32)).tolist() == [1.0] * 4
    assert O.minmax_normalize(np.array([7.0], dtype=F32)).tolist() == [1.0]


def test_minmax_of_a_shard_with_the_scene_range():
    # a shard normalised with the scene's min and max gives, tile for tile, the scene's u: the
    # per-scene min-max (Section 2.3 Stage 1) needs only those two numbers from other shards
    rng = np.random.default_rng(9)
    s = rng.standard_normal(37).astype(F32)
    u = O.minmax_normalize(s)
    for a, b in [(0, 12), (12, 25), (25, 37), (3, 4)]:
        part = O.minmax_normalize(s[a:b], lo=s.min(), hi=s.max())
        assert part.view(np.uint32).tolist() == u[a:b].view(np.uint32).tolist()
    # the shard's own range is the default; a range with max = min gives u = 1
    assert O.minmax_normalize(s, lo=s.min(), hi=s.max()).tolist() == u.tolist()
    assert O.minmax_normalize(s[:3], lo=0.5, hi=0.5).tolist() == [1.0] * 3
    with pytest.raises(O.OracleError):
        O.minmax_normalize(s, lo=np.nan, hi=1.0)


def test_threshold_is_greater_or_equal():
    # u = 0.37f exactly must be kept (Appendix B: u_i >= 0.37; Listing 1: >=)
    s = np.array([0.0, F32(0.37), 1.0], dtype=F32)
    u = O.minmax_normalize(s)
    assert u[1] == F32(0.37)
    assert O.retained(u, 0.37) == [1, 2]
    assert O.retained(np.array([np.nextafter(F32(0.37), F32(0))], dtype=F32), 0.37) == []


def test_nonfinite_scores_raise():
    with pytest.raises(O.OracleError):
        O.minmax_normalize(np.array([0.0, np.nan], dtype=F32))
    with pytest.raises(O.OracleError):
        O.top_b(np.array([0.0, np.inf], dtype=F32), 1)


# ---------------------------------------------------------------- Eq. 2 budget rule (Stage 2)

def _exact_argmax(p: Fraction, pol):
    """Eq. 2 in exact rational arithmetic; returns (budget, margin to the runner-up)."""
    lam = Fraction(str(pol.lam))
    U = [p * Fraction(str(a)) + (1 - p) * Fraction(str(b)) - lam * Fraction(str(e))
         for a, b, e in zip(pol.alpha_pos, pol.alpha_neg, pol.energy)]
    order = sorted(range(len(U)), key=lambda k: (-U[k], k))
    margin = U[order[0]] - U[order[1]] if len(U) > 1 else Fraction(1)
    return pol.C[order[0]], margin


@pytest.mark.parametrize("pol", [W.RIFT_POLICY, W.RIFT_POLICY_SKEW])
def test_budget_truth_table_against_exact_arithmetic(pol):
    for k in range(0, 101):
        p32 = F32(k / 100)
        b_exact, margin = _exact_argmax(Fraction(float(p32)), pol)
        if margin > Fraction(1, 10 ** 5):  # fp32 rounding (~1e-7) cannot flip it
            assert O.budget(float(p32), pol) == b_exact, (k, b_exact)


def test_budget_walkthrough_inversion():
    # Appendix B Step 4: confident (object) tiles get 72 tokens, low-p clutter tiles 288
    pol = W.RIFT_POLICY
    assert O.budget(1.0, pol) == 72
    for p in (0.0, 0.2, 0.37, 0.5, 0.7):
        assert O.budget(p, pol) == 288
    # the skewed policy reaches every budget of C as p grows
    got = {O.budget(k / 100, W.RIFT_POLICY_SKEW) for k in range(101)}
    assert got == set(W.RIFT_POLICY_SKEW.C)


def test_budget_ties_go_to_the_cheaper_budget():
    pol = W.Policy(tau=0.37, C=(72, 144, 288), alpha_pos=(0.5, 0.5, 0.5), alpha_neg=(0.5, 0.5, 0.5),
                   energy=(0.0, 0.0, 0.0), lam=0.0)
    assert O.budget(0.3, pol) == 72


# ---------------------------------------------------------------- top-b (Stage 2: dominant tokens)

@pytest.mark.parametrize("seed", range(8))
def test_top_b_brute_force_with_ties(seed):
    rng = np.random.default_rng(100 + seed)
    n = 9
    r = (rng.integers(-2, 3, size=n) * 0.25).astype(F32)
    r[rng.integers(0, n)] = F32(-0.0)
    r[rng.integers(0, n)] = F32(0.0)
    for b in range(1, n + 1):
        got = O.top_b(r, b)
        assert got == sorted(got) and len(got) == b
        chosen = set(got)
        rest = [k for k in range(n) if k not in chosen]
        for a in chosen:
            for c in rest:  # every selected token beats every unselected one
                assert r[a] > r[c] or (r[a] == r[c] and a < c)


def test_top_b_full_budget_keeps_everything():
    r = np.random.default_rng(0).standard_normal(576).astype(F32)
    assert O.top_b(r, 576) == list(range(576))


# ---------------------------------------------------------------- packing accounting

def test_pack_accounting_and_full_budget_equals_exhaustive():
    wl = W.TINY
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    # full budget on all tiles: tau = 0 keeps every tile, C = {576} keeps every token
    sel = O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, W.KEEP_ALL)
    assert sel.kept == list(range(wl.scene.N))
    assert all(s == list(range(576)) for s in sel.sel)
    H0, cu, pos = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    S, Q = wl.scene.S, wl.scene.Q
    L = S + 576 + Q
    assert cu == [L * i for i in range(wl.scene.N + 1)]
    assert pos == list(range(L)) * wl.scene.N
    for i in range(wl.scene.N):
        exhaustive = torch.cat([sc.embed[sc.sys_ids], sc.X[i].to(torch.bfloat16), sc.embed[sc.query_ids]])
        assert torch.equal(H0[cu[i]:cu[i + 1]], exhaustive)


def test_pack_ragged_accounting():
    wl = W.TINY
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    sel = O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy)
    H0, cu, pos = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    S, Q = wl.scene.S, wl.scene.Q
    assert cu[-1] == H0.shape[0] == sum(S + b + Q for b in sel.budgets)
    assert all(b in wl.policy.C for b in sel.budgets)
    assert [len(s) for s in sel.sel] == sel.budgets
    for j, (i, idx) in enumerate(zip(sel.kept, sel.sel)):
        rows = H0[cu[j]:cu[j + 1]]
        assert torch.equal(rows[S:S + len(idx)], sc.X[i][idx].to(torch.bfloat16))
        assert pos[cu[j]:cu[j + 1]] == list(range(cu[j + 1] - cu[j]))


# ---------------------------------------------------------------- decoder prefill (Section 2.1)

def _tiny_layers(dec, seed=0):
    return [W.make_layer(dec, l, "cpu", seed) for l in range(dec.n_layers)], W.make_final_norm(dec, "cpu", seed)


def _textbook_prefill(H0, layers, g_final, dec):
    """Second, independent formulation: torch SDPA (is_causal), complex-number RoPE,
    F.rms_norm and F.silu, all in fp64."""
    h = H0.to(torch.float64)
    L = h.shape[0]
    hd, H = dec.head_dim, dec.n_heads
    half = hd // 2
    freqs = 1.0 / (dec.rope_theta ** (torch.arange(0, hd, 2, dtype=torch.float64) / hd))
    rot = torch.polar(torch.ones(L, half, dtype=torch.float64), torch.outer(torch.arange(L, dtype=torch.float64), freqs))

    def rope(x):  # x [L, H, hd]; pairs (j, j + hd/2) as one complex number
        z = torch.complex(x[..., :half], x[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    for Wl in layers:
        f = {k: v.to(torch.float64) for k, v in Wl.items()}
        x = F.rms_norm(h, (dec.d,), f["g_attn"], dec.eps)
        q = rope((x @ f["wq"].T).view(L, H, hd)).transpose(0, 1)
        k = rope((x @ f["wk"].T).view(L, H, hd)).transpose(0, 1)
        v = (x @ f["wv"].T).view(L, H, hd).transpose(0, 1)
        a = F.scaled_dot_product_attention(q, k, v, is_causal=True).transpose(0, 1).reshape(L, dec.d)
        h = h + a @ f["wo"].T
        x = F.rms_norm(h, (dec.d,), f["g_ffn"], dec.eps)
        h = h + (F.silu(x @ f["wg"].T) * (x @ f["wu"].T)) @ f["wd"].T
    return F.rms_norm(h, (dec.d,), g_final.to(torch.float64), dec.eps)


def test_prefill_matches_textbook_formulation():
    dec = W.TINY_DECODER
    layers, gf = _tiny_layers(dec)
    H0 = (torch.randn(37, dec.d, generator=torch.Generator().manual_seed(0))).to(torch.bfloat16)
    out = O.prefill_sequence(H0, lambda l: layers[l], gf, dec)
    ref = _textbook_prefill(H0, layers, gf, dec)
    assert torch.allclose(out, ref, rtol=0, atol=1e-10)


def test_prefill_single_token_closed_form():
    # L = 1: softmax over one key is 1 and RoPE at position 0 is the identity, so each layer is
    # h += W_o W_v x then the SwiGLU FFN.
    dec = W.TINY_DECODER
    layers, gf = _tiny_layers(dec)
    h = torch.randn(1, dec.d, generator=torch.Generator().manual_seed(1), dtype=torch.float64)
    ref = h.clone()
    for Wl in layers:
        f = {k: v.to(torch.float64) for k, v in Wl.items()}
        x = ref / torch.sqrt((ref ** 2).mean() + dec.eps) * f["g_attn"]
        ref = ref + (x @ f["wv"].T) @ f["wo"].T
        x = ref / torch.sqrt((ref ** 2).mean() + dec.eps) * f["g_ffn"]
        g = x @ f["wg"].T
        ref = ref + ((g / (1 + torch.exp(-g))) * (x @ f["wu"].T)) @ f["wd"].T
    ref = ref / torch.sqrt((ref ** 2).mean() + dec.eps) * gf.to(torch.float64)
    out = O.prefill_sequence(h, lambda l: layers[l], gf, dec)
    assert torch.allclose(out, ref, rtol=0, atol=1e-12)


def test_prefill_is_causal():
    dec = W.TINY_DECODER
    layers, gf = _tiny_layers(dec)
    H0 = torch.randn(20, dec.d, generator=torch.Generator().manual_seed(2), dtype=torch.float64)
    full = O.prefill_sequence(H0, lambda l: layers[l], gf, dec)
    prefix = O.prefill_sequence(H0[:12], lambda l: layers[l], gf, dec)
    assert torch.allclose(full[:12], prefix, rtol=0, atol=1e-12)
    H1 = H0.clone()
    H1[15] += 1.0
    changed = O.prefill_sequence(H1, lambda l: layers[l], gf, dec)
    assert torch.allclose(changed[:15], full[:15], rtol=0, atol=1e-12)
    assert not torch.allclose(changed[15:], full[15:])


def test_rope_rotation_preserves_norm_and_relative_position():
    x = torch.randn(5, 2, 64, generator=torch.Generator().manual_seed(3), dtype=torch.float64)
    y = O.rope(x, torch.arange(5), 1e4)
    assert torch.allclose(x.norm(dim=-1), y.norm(dim=-1), atol=1e-12)
    assert torch.allclose(O.rope(x, torch.zeros(5, dtype=torch.long), 1e4), x, atol=0)
    # <R(p) a, R(q) b> depends on q - p only
    a, b = x[0, 0], x[1, 0]
    d1 = O.rope(a.view(1, 1, 64), torch.tensor([3]), 1e4).flatten() @ O.rope(b.view(1, 1, 64), torch.tensor([7]), 1e4).flatten()
    d2 = O.rope(a.view(1, 1, 64), torch.tensor([10]), 1e4).flatten() @ O.rope(b.view(1, 1, 64), torch.tensor([14]), 1e4).flatten()
    assert float(d1) == pytest.approx(float(d2), abs=1e-12)


def test_attention_matches_sdpa():
    q, k, v = (torch.randn(13, 3, 16, generator=torch.Generator().manual_seed(s), dtype=torch.float64) for s in (4, 5, 6))
    ref = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                         is_causal=True).transpose(0, 1)
    assert torch.allclose(O.causal_attention(q, k, v), ref, atol=1e-13)


# ------------------------------------------- KV cache, logits and the decode step (Section 2.1)

def _textbook_prefill_kv(H0, layers, dec):
    """The textbook formulation above, also returning each layer's keys (complex-number RoPE)
    and values as [L, d]."""
    h = H0.to(torch.float64)
    L = h.shape[0]
    hd, H = dec.head_dim, dec.n_heads
    half = hd // 2
    freqs = 1.0 / (dec.rope_theta ** (torch.arange(0, hd, 2, dtype=torch.float64) / hd))
    rot = torch.polar(torch.ones(L, half, dtype=torch.float64), torch.outer(torch.arange(L, dtype=torch.float64), freqs))

    def rope(x):
        z = torch.complex(x[..., :half], x[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    cache = []
    for Wl in layers:
        f = {k: v.to(torch.float64) for k, v in Wl.items()}
        x = F.rms_norm(h, (dec.d,), f["g_attn"], dec.eps)
        q = rope((x @ f["wq"].T).view(L, H, hd))
        k = rope((x @ f["wk"].T).view(L, H, hd))
        v = (x @ f["wv"].T).view(L, H, hd)
        cache.append((k.reshape(L, dec.d), v.reshape(L, dec.d)))
        a = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           is_causal=True).transpose(0, 1).reshape(L, dec.d)
        h = h + a @ f["wo"].T
        x = F.rms_norm(h, (dec.d,), f["g_ffn"], dec.eps)
        h = h + (F.silu(x @ f["wg"].T) * (x @ f["wu"].T)) @ f["wd"].T
    return cache


def test_cached_prefill_matches_textbook_hidden_states_and_cache():
    dec = W.TINY_DECODER
    layers, gf = _tiny_layers(dec)
    H0 = (torch.randn(23, dec.d, generator=torch.Generator().manual_seed(7))).to(torch.bfloat16)
    out, cache = O.prefill_with_cache(H0, lambda l: layers[l], gf, dec)
    assert torch.allclose(out, _textbook_prefill(H0, layers, gf, dec), rtol=0, atol=1e-10)
    ref = _textbook_prefill_kv(H0, layers, dec)
    assert len(cache) == dec.n_layers
    for (k, v), (rk, rv) in zip(cache, ref):
        assert k.shape == (23, dec.d) and v.shape == (23, dec.d)
        assert torch.allclose(k, rk, rtol=0, atol=1e-12)
        assert torch.allclose(v, rv, rtol=0, atol=1e-12)


def test_decode_after_prefill_equals_the_longer_prefill():
    # Prefill of L - 1 tokens, then one decode step with token L - 1, must give the same final
    # hidden state and the same new cache rows as prefilling all L tokens at once: catches a
    # wrong decode position, a dropped or duplicated cached row, or the new key left unrotated.
    dec = W.TINY_DECODER
    layers, gf = _tiny_layers(dec)
    H0 = torch.randn(17, dec.d, generator=torch.Generator().manual_seed(8), dtype=torch.float64)
    full, full_cache = O.prefill_with_cache(H0, lambda l: layers[l], gf, dec)
    _, cache = O.prefill_with_cache(H0[:16], lambda l: layers[l], gf, dec)
    h, new = O.decode_token(H0[16], cache, lambda l: layers[l], gf, dec)
    assert torch.allclose(h, full[16], rtol=0, atol=1e-12)
    for (k, v), (fk, fv) in zip(new, full_cache):
        assert torch.allclose(k, fk[16], rtol=0, atol=1e-12)
        assert torch.allclose(v, fv[16], rtol=0, atol=1e-12)


def test_decode_of_the_second_token_by_hand():
    # One layer, P = 1 cached row: the new row's attention is the 2-key softmax written out.
    dec = W.DecoderShape(n_layers=1, d=64, n_heads=2, head_dim=32, ffn=96, vocab=50)
    layers, gf = _tiny_layers(dec, seed=3)
    f = {k: v.to(torch.float64) for k, v in layers[0].items()}
    x0, x1 = torch.randn(2, dec.d, generator=torch.Generator().manual_seed(9), dtype=torch.float64)
    _, cache = O.prefill_with_cache(x0[None], lambda l: layers[l], gf, dec)
    h, _ = O.decode_token(x1, cache, lambda l: layers[l], gf, dec)

    def nrm(v, g):
        return v / math.sqrt(float((v * v).mean()) + dec.eps) * g

    def rot(u, p):  # rotate-half RoPE of one head vector at position p
        half = u.shape[0] // 2
        ang = p * dec.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / u.shape[0])
        return torch.cat([u[:half] * torch.cos(ang) - u[half:] * torch.sin(ang),
                          u[half:] * torch.cos(ang) + u[:half] * torch.sin(ang)])

    a0, a1 = nrm(x0, f["g_attn"]), nrm(x1, f["g_attn"])
    att = []
    for hh in range(dec.n_heads):
        sl = slice(hh * 32, hh * 32 + 32)
        q = rot((f["wq"] @ a1)[sl], 1)
        k0, k1 = (f["wk"] @ a0)[sl], rot((f["wk"] @ a1)[sl], 1)
        v0, v1 = (f["wv"] @ a0)[sl], (f["wv"] @ a1)[sl]
        s0, s1 = float(q @ k0) / math.sqrt(32), float(q @ k1) / math.sqrt(32)
        w0 = 1.0 / (1.0 + math.exp(s1 - s0))
        att.append(w0 * v0 + (1.0 - w0) * v1)
    r = x1 + f["wo"] @ torch.cat(att)
    y = nrm(r, f["g_ffn"])
    g = f["wg"] @ y
    r = r + f["wd"] @ ((g / (1.0 + torch.exp(-g))) * (f["wu"] @ y))
    assert torch.allclose(h, nrm(r, gf.to(torch.float64)), rtol=0, atol=1e-12)


def test_attention_with_past_matches_masked_sdpa():
    q = torch.randn(4, 3, 16, generator=torch.Generator().manual_seed(10), dtype=torch.float64)
    k, v = (torch.randn(11, 3, 16, generator=torch.Generator().manual_seed(s), dtype=torch.float64) for s in (11, 12))
    allowed = torch.arange(11)[None, :] <= (7 + torch.arange(4))[:, None]
    ref = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                         attn_mask=allowed).transpose(0, 1)
    assert torch.allclose(O.attention_with_past(q, k, v, 7), ref, atol=1e-13)
    assert torch.allclose(O.attention_with_past(q, k[:4], v[:4], 0), O.causal_attention(q, k[:4], v[:4]), atol=1e-14)


def test_logits_select_rows_of_the_output_matrix():
    # A permutation output matrix picks hidden coordinates: logits[r] = h[perm[r]]; a transposed
    # operand would give h[perm^-1[r]] instead.
    d = 12
    perm = torch.randperm(d, generator=torch.Generator().manual_seed(13))
    W_lm = torch.zeros(d, d, dtype=torch.float64)
    W_lm[torch.arange(d), perm] = 1.0
    h = torch.randn(3, d, generator=torch.Generator().manual_seed(14), dtype=torch.float64)
    assert torch.equal(O.logits(h, W_lm), h[:, perm])
    assert not torch.equal(h[:, perm], h[:, torch.argsort(perm)])
    W2 = torch.randn(5, d, generator=torch.Generator().manual_seed(15), dtype=torch.float64)
    assert torch.allclose(O.logits(h[0], W2), torch.stack([W2[r] @ h[0] for r in range(5)]), atol=1e-14)


# ------------------------------------- contextual-token merge (Stage 2: VisionZip's mechanism)

def test_contextual_count_matches_visionzip_splits():
    P = W.RIFT_POLICY_MERGE
    # VisionZip's LLaVA-1.5 settings: 64 = 54 + 10, 128 = 108 + 20, 192 = 162 + 30 tokens
    assert [O.contextual_count(c, 576, P) for c in (64, 128, 192)] == [10, 20, 30]
    assert O.contextual_count(576, 576, P) == 0              # full budget: nothing left to merge
    assert O.contextual_count(288, 576, W.RIFT_POLICY) == 0  # merge off
    assert [O.contextual_count(c, 576, P) for c in P.C] == [11, 22, 45, 67, 0]


def _rest(n_v, dominant):
    return [k for k in range(n_v) if k not in set(dominant)]


def test_merge_recovers_planted_clusters():
    # 12 remaining tokens (dominant ones interleaved) in 3 tight clusters of 4 consecutive
    # remaining tokens around orthogonal directions.  With m = 3 the targets are the 1st, 5th and
    # 9th remaining tokens, one per cluster, so the groups are the clusters and each contextual
    # token is its cluster's mean.  A target step taken over all tokens instead of the remaining
    # ones, or an off-by-one, puts two targets in one cluster.
    g = torch.Generator().manual_seed(20)
    n_v, d = 15, 6
    dominant = [1, 5, 9]
    rest = _rest(n_v, dominant)
    X = 0.01 * torch.randn(n_v, d, generator=g, dtype=torch.float64)
    for c in range(3):
        for k in rest[4 * c:4 * c + 4]:
            X[k, 2 * c] += 1.0 + 0.1 * c
    targets, groups, ctx = O.merge_contextual(X, dominant, 3)
    assert targets == [rest[0], rest[4], rest[8]]
    assert [sorted(gr) for gr in groups] == [rest[0:4], rest[4:8], rest[8:12]]
    for c in range(3):
        assert torch.allclose(ctx[c], X[rest[4 * c:4 * c + 4]].mean(dim=0), atol=1e-15)


def test_merge_special_cases():
    g = torch.Generator().manual_seed(21)
    X = torch.randn(10, 4, generator=g, dtype=torch.float64)
    dominant = [2, 7]
    rest = _rest(10, dominant)
    t, gr, ctx = O.merge_contextual(X, dominant, len(rest))    # every remaining token a target
    assert t == rest and torch.equal(ctx, X[rest])
    t, gr, ctx = O.merge_contextual(X, dominant, 1)            # one target takes everything
    assert t == [rest[0]] and torch.allclose(ctx[0], X[rest].mean(dim=0), atol=1e-15)
    assert O.merge_contextual(X, dominant, 0)[2].shape == (0, 4)
    assert O.merge_contextual(X, list(range(10)), 3)[2].shape == (0, 4)   # nothing left
    assert O.merge_contextual(X, dominant, 50)[0] == rest                 # m capped at R


@pytest.mark.parametrize("seed", [22, 23, 24])
def test_merge_assignment_brute_force_cosine(seed):
    g = torch.Generator().manual_seed(seed)
    n_v, d, m = 30, 8, 5
    X = torch.randn(n_v, d, generator=g, dtype=torch.float64)
    dominant = sorted(torch.randperm(n_v, generator=g)[:7].tolist())
    rest = _rest(n_v, dominant)
    targets, groups, _ = O.merge_contextual(X, dominant, m)
    step = len(rest) // m
    assert targets == rest[::step][:m]
    owner = {k: j for j, gr in enumerate(groups) for k in gr}
    for k in rest:
        if k in targets:
            assert owner[k] == targets.index(k)
            continue
        sims = [1.0 - distance.cosine(X[k].numpy(), X[t].numpy()) for t in targets]
        best = max(range(m), key=lambda j: (sims[j], -j))
        assert owner[k] == best
    # scale invariance of the assignment (positive factors on the non-target tokens)
    Xs = X.clone()
    for k in rest:
        if k not in targets:
            Xs[k] *= 0.5 + k
    assert O.merge_contextual(Xs, dominant, m)[1] == groups


def test_merge_ties_go_to_the_lower_target_and_mass_is_conserved():
    # every token points the same way, so all four targets (0, 2, 4, 6) tie for every token
    X = torch.zeros(8, 3, dtype=torch.float64)
    X[:, 0] = torch.arange(1, 9, dtype=torch.float64)
    _, groups, ctx = O.merge_contextual(X, [], 4)
    assert groups == [[0, 1, 3, 5, 7], [2], [4], [6]]
    g = torch.Generator().manual_seed(25)
    Y = torch.randn(40, 6, generator=g, dtype=torch.float64)
    dominant = [0, 3, 17, 39]
    rest = _rest(40, dominant)
    _, groups, ctx = O.merge_contextual(Y, dominant, 6)
    assert sorted(k for gr in groups for k in gr) == rest
    total = sum(len(gr) * ctx[j] for j, gr in enumerate(groups))
    assert torch.allclose(total, Y[rest].sum(dim=0), atol=1e-12)


def test_selection_with_merge_splits_every_budget():
    from dataclasses import replace
    wl = replace(W.TINY, policy=replace(W.TINY.policy, ctx_num=10, ctx_den=64))
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    sel = O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy)
    n_v = wl.scene.n_v
    for i, idx, b, ctx in zip(sel.kept, sel.sel, sel.budgets, sel.ctx):
        m = O.contextual_count(b, n_v, wl.policy)
        assert len(idx) == b - m and ctx.shape[0] == m
        assert idx == O.top_b(sel.r32[i], b - m)
    H0, cu, pos = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids, sel.ctx)
    S, Q = wl.scene.S, wl.scene.Q
    assert [cu[j + 1] - cu[j] for j in range(len(sel.kept))] == [S + b + Q for b in sel.budgets]
    for j, (i, idx, ctx) in enumerate(zip(sel.kept, sel.sel, sel.ctx)):
        a = cu[j] + S
        assert torch.equal(H0[a:a + len(idx)], sc.X[i][idx].to(torch.bfloat16))
        assert torch.equal(H0[a + len(idx):a + len(idx) + ctx.shape[0]], ctx.to(torch.bfloat16))


# ------------------------------- predictor features (Section 2.3, Stage 2: quadrant scores)

def _tq(d=16, M=3, seed=30):
    g = torch.Generator().manual_seed(seed)
    t = O.l2norm(torch.randn(d, generator=g, dtype=torch.float64))
    B = torch.stack([O.l2norm(torch.randn(d, generator=g, dtype=torch.float64)) for _ in range(M)])
    return t, B


def test_quadrants_of_a_uniform_tile_equal_the_tile_score():
    t, B = _tq()
    row = torch.randn(16, generator=torch.Generator().manual_seed(31), dtype=torch.float64)
    X = row.repeat(36, 1)  # 6 x 6 grid, every token the same
    q = O.quadrant_scores(X, t, B)
    s = O.margin(O.tile_embedding(X)[None, :], t, B)[0]
    assert torch.allclose(q, s.expand(4), atol=1e-14)


def test_quadrants_partition_the_grid_and_follow_a_planted_patch():
    t, B = _tq()
    g = torch.Generator().manual_seed(32)
    X = torch.randn(64, 16, generator=g, dtype=torch.float64)  # 8 x 8 grid
    # the pooled tile sum is the sum of the four quadrant sums: every token in exactly one quadrant
    grid = X.view(8, 8, 16)
    qs = [grid[:4, :4], grid[:4, 4:], grid[4:, :4], grid[4:, 4:]]
    assert torch.allclose(sum(q.reshape(-1, 16).sum(0) for q in qs), X.sum(0), atol=1e-12)
    # plant the query direction on a patch inside the bottom-right quadrant (rows 5-6, cols 5-7)
    for r in (5, 6):
        for c in (5, 6, 7):
            X[r * 8 + c] += 6.0 * t
    q = O.quadrant_scores(X, t, B)
    assert int(torch.argmax(q)) == 3
    # a left-right mirror of the grid swaps top-left/top-right and bottom-left/bottom-right
    Xm = X.view(8, 8, 16).flip(1).reshape(64, 16)
    assert torch.allclose(O.quadrant_scores(Xm, t, B), q[[1, 0, 3, 2]], atol=1e-14)
    with pytest.raises(O.OracleError):
        O.quadrant_scores(X[:63], t, B)


def test_token_stats_match_numpy():
    r = np.random.default_rng(33).standard_normal(576).astype(np.float32)
    mx, mean, std = O.token_stats(r)
    r64 = r.astype(np.float64)
    assert mx == float(r64.max()) and mean == pytest.approx(float(r64.mean()), abs=1e-15)
    assert std == pytest.approx(float(r64.std()), abs=1e-14)


def test_suffix_over_a_shared_prefix_equals_the_whole_prefill():
    # The prefix (system prompt) prefilled once and each sequence's suffix extended from its
    # cache give the whole sequence's prefill: same suffix hidden states and cache rows.
    dec = W.TINY_DECODER
    layers, gf = _tiny_layers(dec)
    g = torch.Generator().manual_seed(34)
    prefix = torch.randn(8, dec.d, generator=g, dtype=torch.float64)
    pre_h, pre_cache = O.prefill_with_cache(prefix, lambda l: layers[l], gf, dec)
    for n in (1, 5, 13):
        suffix = torch.randn(n, dec.d, generator=g, dtype=torch.float64)
        full, full_cache = O.prefill_with_cache(torch.cat([prefix, suffix]), lambda l: layers[l], gf, dec)
        h, new = O.extend_with_cache(suffix, pre_cache, lambda l: layers[l], gf, dec)
        assert torch.allclose(full[:8], pre_h, rtol=0, atol=1e-12)
        assert torch.allclose(full[8:], h, rtol=0, atol=1e-12)
        for (k, v), (fk, fv) in zip(new, full_cache):
            assert torch.allclose(k, fk[8:], rtol=0, atol=1e-12) and torch.allclose(v, fv[8:], rtol=0, atol=1e-12)
    # the one-row case is the decode step
    x = torch.randn(dec.d, generator=g, dtype=torch.float64)
    h1, _ = O.extend_with_cache(x[None], pre_cache, lambda l: layers[l], gf, dec)
    h2, _ = O.decode_token(x, pre_cache, lambda l: layers[l], gf, dec)
    assert torch.equal(h1[0], h2)
