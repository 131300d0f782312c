"""Plain, slow CPU oracle for Rift's hot path (tile pruning + elastic prefill).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import or run this module.  It shares no
code with the CUDA library and never imports it.

Each function restates one step of the paper in the paper's order:

  Section 2.3, Stage 1, Eq. 1 ......... background-margin relevance s_i
  Appendix B, Step 2 / Listing 1 ...... kNN smoothing (m = 6), per-scene min-max
  Appendix B, Step 3 / Listing 1 ...... retain tiles with u_i >= tau (tau = 0.37)
  Section 2.3, Stage 2, Eq. 2 ......... U_i(c) = A_i(c) - lambda E_c,
                                         A_i(c) = p_i a+_c + (1 - p_i) a-_c, c* = argmax
  Section 2.3, Stage 2 ................ keep each retained tile's dominant tokens and merge
                                         the remainder into contextual tokens (VisionZip)
  Section 2.1 ......................... decoder prefill over [system | vision | query],
                                         the KV cache it builds, the last-token logits
                                         and the decode step that follows it

Precision.  Scores are computed in fp64 and rounded once to fp32; every
decision (min-max, threshold, utility argmax, top-b order) is then taken in
fp32, with each fp32 operation written out one at a time in the order given
below, so the result is fixed by IEEE round-to-nearest.  The one exception is
the neighbour choice of the smoothing step: tile similarities are compared in
fp64, because nearly parallel tiles have similarities closer to 1 than fp32's
spacing there (6e-8), which would turn their order into a rounding accident.
The prefill is fp64 throughout, on weights and inputs that are bf16 values.

Readings of points the paper leaves open (each also used by the CUDA path):
  * Stand-in embeddings (the paper uses RemoteCLIP): V_i = l2norm(mean_k x_ik)
    over tile i's projected tokens; t = l2norm of the mean embedding row of the
    query ids (with several caption templates, t = l2norm(mean_k l2norm(e_k)));
    B_j = l2norm(embedding row of background id j).
  * Token ranking: Eq. 1 applied to each vision token, r_ik = x^_ik t -
    mean_j x^_ik B_j, with x^ = x / ||x||.
  * Smoothing: cosine similarity G = V V^T, self excluded, the m = min(6, N-1)
    most similar tiles (ties to the lower index), unweighted mean with self of
    the raw scores, one pass.  The fp32 sum runs over the set {i} + NN(i) in
    ascending tile index, then divides by m + 1, so tiles whose sets are equal
    get bit-equal smoothed scores (with m = N - 1 every set is the whole scene
    and every u is 1, as the exact arithmetic says).
  * Threshold is ">=" (Appendix B and Listing 1).  If max = min, u = 1 for all.
  * Utility in fp32 as ((p * a+) + ((1 - p) * a-)) - (lambda * E); C ascending,
    ties to the lower index (the cheaper budget).
  * Top-b: the b largest r, ties to the lower token index, listed ascending.
  * Merge (policy ctx_num > 0; the paper uses VisionZip's mechanism without details): a budget
    c < n_v holds m = floor(ctx_num c / ctx_den) contextual tokens and c - m dominant ones.  Of
    the R tokens not selected (ascending), every floor(R / m)-th from the first is a target;
    every other one joins the target with the largest cosine similarity (ties to the lower
    target), in the projected-token space (the paper's encoder keys are not available); a
    contextual token is the mean of its group, target included.  Sequence i = [S system ids |
    c - m dominant tokens | m contextual tokens in target order | Q query ids].
  * Sequence i = [S system ids | b_i selected tokens | Q query ids], positions
    0 .. L_i - 1, tiles in ascending index order.
  * Decoder: LLaMA block, RMSNorm (eps 1e-6), rotate-half RoPE (theta 1e4),
    causal softmax attention with scale 1/sqrt(head_dim), SwiGLU, final RMSNorm.
  * KV cache: per layer, the keys after RoPE and the values, [L, H * head_dim]
    with heads contiguous.  Logits: final hidden state of a sequence's last
    token times the untied output matrix, [vocab, d].  Decode: one new token
    per sequence at position L_i (the next after its prompt), attending to the
    cached keys and values of its own sequence and to itself.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch

F32 = np.float32


class OracleError(ValueError):
    pass


# ------------------------------------------------------------------------------------------
# a1  Query preparation (Stage 1: "embed the query's object of interest and a fixed vocabulary
#     of background terms", stand-in C1)
# ------------------------------------------------------------------------------------------

def l2norm(v: torch.Tensor) -> torch.Tensor:
    v = v.to(torch.float64)
    return v / torch.sqrt((v * v).sum(dim=-1, keepdim=True))


def query_embedding(embed: torch.Tensor, phrase_ids) -> torch.Tensor:
    """t for one query.  ``phrase_ids`` is a list of id lists, one per caption template."""
    if phrase_ids and isinstance(phrase_ids[0], int):
        phrase_ids = [phrase_ids]
    e = [embed[list(ids)].to(torch.float64).mean(dim=0) for ids in phrase_ids]
    return l2norm(torch.stack([l2norm(x) for x in e]).mean(dim=0))


def background_embeddings(embed: torch.Tensor, bg_ids) -> torch.Tensor:
    """B [M, d]; M = 0 gives an empty [0, d] matrix."""
    if len(bg_ids) == 0:
        return torch.zeros(0, embed.shape[1], dtype=torch.float64)
    return l2norm(embed[list(bg_ids)].to(torch.float64))


# ------------------------------------------------------------------------------------------
# a2 / a3  Eq. 1 on tokens and on tiles
# ------------------------------------------------------------------------------------------

def margin(U: torch.Tensor, t: torch.Tensor, B: torch.Tensor) -> torch.Tensor:
    """Eq. 1 written out: U t - (1/M) sum_j U B_j^T for unit rows U (fp64).  M = 0 drops the
    background term."""
    s = U @ t
    if B.shape[0] > 0:
        s = s - (U @ B.T).mean(dim=1)
    return s


def token_relevance(X_tile: torch.Tensor, t, B) -> torch.Tensor:
    """r_ik for the n_v tokens of one tile (fp64)."""
    return margin(l2norm(X_tile), t, B)


def tile_embedding(X_tile: torch.Tensor) -> torch.Tensor:
    """V_i = l2norm(mean of the tile's tokens) (fp64)."""
    return l2norm(X_tile.to(torch.float64).mean(dim=0))


def score_scene(X: torch.Tensor, t, B):
    """Per tile: fp64 token scores r [N, n_v], embeddings V [N, d], Eq. 1 scores s [N]."""
    N = X.shape[0]
    r = torch.empty(N, X.shape[1], dtype=torch.float64)
    V = torch.empty(N, X.shape[2], dtype=torch.float64)
    for i in range(N):
        xi = X[i].to(torch.float64)
        r[i] = token_relevance(xi, t, B)
        V[i] = tile_embedding(xi)
    s = margin(V, t, B)
    return r, V, s


def to_f32(x) -> np.ndarray:
    if isinstance(x, torch.Tensor):
        x = x.to(torch.float64).numpy()
    return np.asarray(x, dtype=np.float64).astype(F32)


def quadrant_scores(X_tile: torch.Tensor, t, B) -> torch.Tensor:
    """Eq. 1 of the four quadrants of the tile's token grid (Section 2.3, Stage 2: a predictor
    feature): tokens k = row * g + col of the g x g grid (n_v = g^2, g even) split into rows
    < g/2 or not and columns < g/2 or not; quadrant order top-left, top-right, bottom-left,
    bottom-right; each scored as l2norm(mean of its tokens), fp64 [4]."""
    n_v = X_tile.shape[0]
    g = int(round(math.sqrt(n_v)))
    if g * g != n_v or g % 2:
        raise OracleError("quadrants need an even square token grid")
    h = g // 2
    x = X_tile.to(torch.float64).view(g, g, -1)
    quads = [x[:h, :h], x[:h, h:], x[h:, :h], x[h:, h:]]
    V = torch.stack([l2norm(q.reshape(-1, q.shape[-1]).sum(dim=0)) for q in quads])
    return margin(V, t, B)


def token_stats(r_tile) -> tuple:
    """(max, mean, population standard deviation) of a tile's token scores, in fp64."""
    r = np.asarray(r_tile, dtype=np.float64)
    mean = float(r.sum() / r.size)
    return float(r.max()), mean, float(math.sqrt(((r - mean) ** 2).sum() / r.size))


# ------------------------------------------------------------------------------------------
# a4  kNN smoothing (Appendix B Step 2; Listing 1 comment: smoothed with the 6 most similar tiles)
# ------------------------------------------------------------------------------------------

def similarity(V: torch.Tensor) -> np.ndarray:
    """Cosine similarities G = V V^T in fp64 (the neighbour decision compares these)."""
    return (V @ V.T).numpy()


def knn_neighbours(G: np.ndarray, m: int) -> np.ndarray:
    """For each i: the m tiles j != i of largest G_ij, ties to the lower j, in rank order."""
    N = G.shape[0]
    m = min(m, N - 1)
    nbr = np.zeros((N, max(m, 0)), dtype=np.int64)
    for i in range(N):
        cand = [(-float(G[i, j]), j) for j in range(N) if j != i]
        cand.sort()
        nbr[i] = [j for _, j in cand[:m]]
    return nbr


def smooth(s32: np.ndarray, nbr: np.ndarray) -> np.ndarray:
    """s~_i = (s_i + sum_{j in NN(i)} s_j) / (m + 1), fp32, summed over {i} + NN(i) in
    ascending tile index."""
    N, m = nbr.shape if nbr.ndim == 2 else (len(s32), 0)
    out = np.empty(N, dtype=F32)
    div = F32(m + 1)
    for i in range(N):
        members = sorted([i] + [int(j) for j in nbr[i]])
        acc = F32(0.0)
        for j in members:
            acc = F32(acc + F32(s32[j]))
        out[i] = F32(acc / div)
    return out


# ------------------------------------------------------------------------------------------
# a5  per-scene min-max and the threshold (Section 2.3 Stage 1; Appendix B Step 3)
# ------------------------------------------------------------------------------------------

def minmax_normalize(s32: np.ndarray, lo=None, hi=None) -> np.ndarray:
    """u = (s - min) / (max - min) in fp32 over the scene.  lo, hi: the scene's min and max when
    s32 holds only some of its tiles (a shard); by default those of s32 itself."""
    s32 = np.asarray(s32, dtype=F32)
    if not np.all(np.isfinite(s32)):
        raise OracleError("non-finite tile score")
    lo = F32(s32.min()) if lo is None else F32(lo)
    hi = F32(s32.max()) if hi is None else F32(hi)
    if not (np.isfinite(lo) and np.isfinite(hi)):
        raise OracleError("non-finite score range")
    if hi == lo:
        return np.ones_like(s32)
    rng = F32(hi - lo)
    return ((s32 - lo).astype(F32) / rng).astype(F32)


def retained(u32: np.ndarray, tau: float) -> list:
    t = F32(tau)
    return [i for i in range(len(u32)) if u32[i] >= t]


# ------------------------------------------------------------------------------------------
# a6  elastic budget (Eq. 2 and the argmax that follows it)
# ------------------------------------------------------------------------------------------

def utility(p: float, policy) -> list:
    """U(c) for every c in C, in fp32 with the operation order ((p a+) + ((1-p) a-)) - (lam E)."""
    p = F32(p)
    q = F32(F32(1.0) - p)
    lam = F32(policy.lam)
    out = []
    for ap, an, e in zip(policy.alpha_pos, policy.alpha_neg, policy.energy):
        acc = F32(F32(p * F32(ap)) + F32(q * F32(an)))
        out.append(F32(acc - F32(lam * F32(e))))
    return out


def budget(p: float, policy) -> int:
    U = utility(p, policy)
    best = 0
    for k in range(1, len(U)):
        if U[k] > U[best]:
            best = k
    return policy.C[best]


# ------------------------------------------------------------------------------------------
# a7  per-tile top-b (Stage 2: keep the dominant tokens)
# ------------------------------------------------------------------------------------------

def top_b(r32: np.ndarray, b: int) -> list:
    r32 = np.asarray(r32, dtype=F32)
    if not np.all(np.isfinite(r32)):
        raise OracleError("non-finite token score")
    order = sorted(range(len(r32)), key=lambda k: (-float(r32[k]), k))
    return sorted(order[:b])


def contextual_count(c: int, n_v: int, policy) -> int:
    """Contextual tokens inside a budget of c tokens (none at the full budget or without merge)."""
    num = getattr(policy, "ctx_num", 0)
    if num == 0 or c >= n_v:
        return 0
    return (num * c) // policy.ctx_den


def merge_contextual(X_tile: torch.Tensor, dominant, m: int):
    """VisionZip-style merge of the tokens not in `dominant`: (targets, groups, ctx fp64 [m, d]).
    groups[j] lists target j first, then the tokens that joined it in ascending index."""
    n_v, d = X_tile.shape
    keep = set(int(k) for k in dominant)
    rest = [k for k in range(n_v) if k not in keep]
    m = min(m, len(rest))
    if m == 0:
        return [], [], torch.zeros(0, d, dtype=torch.float64)
    step = len(rest) // m
    targets = [rest[j * step] for j in range(m)]
    x = X_tile.to(torch.float64)
    xt = x[targets]
    nrm = torch.sqrt((xt * xt).sum(dim=1, keepdim=True))
    xt_hat = torch.where(nrm > 0, xt / torch.where(nrm > 0, nrm, torch.ones_like(nrm)), torch.zeros_like(xt))
    groups = [[t] for t in targets]
    tset = set(targets)
    for k in rest:
        if k in tset:
            continue
        sim = xt_hat @ x[k]  # cosine up to the positive factor 1 / ||x_k||
        best = 0
        for j in range(1, m):
            if float(sim[j]) > float(sim[best]):
                best = j
        groups[best].append(k)
    ctx = torch.stack([x[g].mean(dim=0) for g in groups])
    return targets, groups, ctx


# ------------------------------------------------------------------------------------------
# a8  packing into per-tile sequences [system | selected vision tokens | query]
# ------------------------------------------------------------------------------------------

def pack(X, embed, kept, sel, sys_ids, query_ids, ctx=None):
    """Returns (H0 bf16 [T, d], cu_seqlens [n+1], positions [T]).  ctx: per kept tile its
    contextual tokens (fp64 [m, d]), placed after the dominant ones."""
    rows, cu, pos = [], [0], []
    sys_rows = embed[list(sys_ids)].to(torch.bfloat16)
    q_rows = embed[list(query_ids)].to(torch.bfloat16)
    for n, (i, idx) in enumerate(zip(kept, sel)):
        vis = X[i][list(idx)].to(torch.bfloat16)
        if ctx is not None and len(ctx[n]):
            vis = torch.cat([vis, ctx[n].to(torch.bfloat16)], dim=0)
        seq = torch.cat([sys_rows, vis, q_rows], dim=0)
        rows.append(seq)
        cu.append(cu[-1] + seq.shape[0])
        pos.extend(range(seq.shape[0]))
    H0 = torch.cat(rows, dim=0) if rows else torch.zeros(0, embed.shape[1], dtype=torch.bfloat16)
    return H0, cu, pos


# ------------------------------------------------------------------------------------------
# a9  decoder prefill (Section 2.1: prefill reads the whole prompt and builds the KV cache)
# ------------------------------------------------------------------------------------------

def rmsnorm(h: torch.Tensor, g: torch.Tensor, eps: float) -> torch.Tensor:
    return h / torch.sqrt((h * h).mean(dim=-1, keepdim=True) + eps) * g.to(torch.float64)


def rope(x: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """Rotate-half RoPE on [L, H, hd]: dims j and j + hd/2 form a pair with frequency
    theta^(-2j/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    j = torch.arange(half, dtype=torch.float64)
    inv = theta ** (-2.0 * j / hd)
    ang = pos.to(torch.float64)[:, None] * inv[None, :]
    c, s = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1)


def causal_attention(q, k, v) -> torch.Tensor:
    """softmax(q k^T / sqrt(hd) + causal mask) v per head; q, k, v: [L, H, hd]."""
    L, H, hd = q.shape
    out = torch.empty_like(q)
    mask = torch.triu(torch.ones(L, L, dtype=torch.bool), diagonal=1)
    for h in range(H):
        sc = (q[:, h] @ k[:, h].T) / math.sqrt(hd)
        sc = sc.masked_fill(mask, float("-inf"))
        sc = sc - sc.max(dim=1, keepdim=True).values
        p = torch.exp(sc)
        p = p / p.sum(dim=1, keepdim=True)
        out[:, h] = p @ v[:, h]
    return out


def silu(x):
    return x / (1.0 + torch.exp(-x))


def decoder_layer(h: torch.Tensor, W: dict, dec, pos: torch.Tensor) -> torch.Tensor:
    L = h.shape[0]
    f = {k: v.to(torch.float64) for k, v in W.items()}
    x = rmsnorm(h, f["g_attn"], dec.eps)
    q = (x @ f["wq"].T).view(L, dec.n_heads, dec.head_dim)
    k = (x @ f["wk"].T).view(L, dec.n_heads, dec.head_dim)
    v = (x @ f["wv"].T).view(L, dec.n_heads, dec.head_dim)
    q, k = rope(q, pos, dec.rope_theta), rope(k, pos, dec.rope_theta)
    a = causal_attention(q, k, v).reshape(L, dec.d)
    h = h + a @ f["wo"].T
    x = rmsnorm(h, f["g_ffn"], dec.eps)
    h = h + (silu(x @ f["wg"].T) * (x @ f["wu"].T)) @ f["wd"].T
    return h


def attention_with_past(q, k, v, n_past: int) -> torch.Tensor:
    """Attention of n new rows (q: [n, H, hd]) over n_past cached rows followed by the new
    rows themselves (k, v: [n_past + n, H, hd]): new row i sees keys 0 .. n_past + i."""
    n, H, hd = q.shape
    P = k.shape[0]
    out = torch.empty_like(q)
    key = torch.arange(P)[None, :]
    mask = key > (n_past + torch.arange(n))[:, None]
    for h in range(H):
        sc = (q[:, h] @ k[:, h].T) / math.sqrt(hd)
        sc = sc.masked_fill(mask, float("-inf"))
        sc = sc - sc.max(dim=1, keepdim=True).values
        p = torch.exp(sc)
        p = p / p.sum(dim=1, keepdim=True)
        out[:, h] = p @ v[:, h]
    return out


def decoder_layer_cached(h: torch.Tensor, W: dict, dec, pos: torch.Tensor, k_past=None, v_past=None):
    """One decoder layer for new rows h at positions pos, given the layer's cached keys (after
    RoPE) and values of the rows before them ([P, H, hd] each, or None).  Returns the new rows'
    hidden states and their keys and values (the rows this layer appends to its cache)."""
    n = h.shape[0]
    f = {k: v.to(torch.float64) for k, v in W.items()}
    x = rmsnorm(h, f["g_attn"], dec.eps)
    q = (x @ f["wq"].T).view(n, dec.n_heads, dec.head_dim)
    k = (x @ f["wk"].T).view(n, dec.n_heads, dec.head_dim)
    v = (x @ f["wv"].T).view(n, dec.n_heads, dec.head_dim)
    q, k = rope(q, pos, dec.rope_theta), rope(k, pos, dec.rope_theta)
    n_past = 0 if k_past is None else k_past.shape[0]
    k_all = k if k_past is None else torch.cat([k_past, k], 0)
    v_all = v if v_past is None else torch.cat([v_past, v], 0)
    a = attention_with_past(q, k_all, v_all, n_past).reshape(n, dec.d)
    h = h + a @ f["wo"].T
    x = rmsnorm(h, f["g_ffn"], dec.eps)
    h = h + (silu(x @ f["wg"].T) * (x @ f["wu"].T)) @ f["wd"].T
    return h, k, v


def prefill_with_cache(H0_seq: torch.Tensor, get_layer, g_final, dec):
    """Prefill of one sequence that also returns the KV cache it builds (Section 2.1): final
    hidden states fp64 [L, d] and, per layer, (keys after RoPE, values) as fp64 [L, d]."""
    h = H0_seq.to(torch.float64)
    pos = torch.arange(h.shape[0])
    cache = []
    for l in range(dec.n_layers):
        h, k, v = decoder_layer_cached(h, get_layer(l), dec, pos)
        cache.append((k.reshape(-1, dec.d), v.reshape(-1, dec.d)))
    return rmsnorm(h, g_final.to(torch.float64), dec.eps), cache


def extend_with_cache(H_new: torch.Tensor, cache, get_layer, g_final, dec):
    """The rows H_new [n, d] appended after the P cached rows of a sequence (positions P ..
    P + n - 1), each attending to the cache and causally to the new rows: their final hidden
    states fp64 [n, d] and, per layer, their (keys after RoPE, values) fp64 [n, d].  With the
    system prompt as the cache this is the prefill of a sequence's suffix over a shared prefix."""
    h = H_new.to(torch.float64)
    P = cache[0][0].shape[0]
    pos = torch.arange(P, P + h.shape[0])
    new = []
    for l in range(dec.n_layers):
        kp = cache[l][0].view(P, dec.n_heads, dec.head_dim)
        vp = cache[l][1].view(P, dec.n_heads, dec.head_dim)
        h, k, v = decoder_layer_cached(h, get_layer(l), dec, pos, kp, vp)
        new.append((k.reshape(-1, dec.d), v.reshape(-1, dec.d)))
    return rmsnorm(h, g_final.to(torch.float64), dec.eps), new


def decode_token(x_emb: torch.Tensor, cache, get_layer, g_final, dec):
    """One decode step of one sequence: the new token's input embedding x_emb [d] at position
    P = len(cache rows), attending to the cached rows and itself.  Returns its final hidden
    state fp64 [d] and, per layer, its (key after RoPE, value) rows fp64 [d]."""
    h = x_emb.to(torch.float64)[None, :]
    P = cache[0][0].shape[0]
    pos = torch.tensor([P])
    new = []
    for l in range(dec.n_layers):
        kp = cache[l][0].view(P, dec.n_heads, dec.head_dim)
        vp = cache[l][1].view(P, dec.n_heads, dec.head_dim)
        h, k, v = decoder_layer_cached(h, get_layer(l), dec, pos, kp, vp)
        new.append((k.reshape(dec.d), v.reshape(dec.d)))
    return rmsnorm(h, g_final.to(torch.float64), dec.eps)[0], new


def logits(h_final: torch.Tensor, W_lm: torch.Tensor) -> torch.Tensor:
    """Output logits of final hidden states h_final [..., d]: h W_lm^T with W_lm [vocab, d]."""
    return h_final.to(torch.float64) @ W_lm.to(torch.float64).T


def prefill_sequence(H0_seq: torch.Tensor, get_layer, g_final, dec) -> torch.Tensor:
    """Final hidden states (after the final RMSNorm) of one sequence, fp64 [L, d].
    ``get_layer(l)`` returns layer l's weights (lets the caller stream 7B layers)."""
    h = H0_seq.to(torch.float64)
    pos = torch.arange(h.shape[0])
    for l in range(dec.n_layers):
        h = decoder_layer(h, get_layer(l), dec, pos)
    return rmsnorm(h, g_final.to(torch.float64), dec.eps)


# ------------------------------------------------------------------------------------------
# The whole selection chain
# ------------------------------------------------------------------------------------------

@dataclass
class Selection:
    t: torch.Tensor
    B: torch.Tensor
    r64: torch.Tensor          # [N, n_v] fp64 token scores
    V: torch.Tensor            # [N, d] fp64 tile embeddings
    s64: torch.Tensor          # [N] fp64 Eq. 1 tile scores
    r32: np.ndarray
    s32: np.ndarray
    G: np.ndarray              # [N, N] fp64 similarities
    nbr: np.ndarray            # [N, m]
    s_tilde: np.ndarray        # [N] fp32
    u: np.ndarray              # [N] fp32
    kept: list
    p: np.ndarray              # [n_kept] fp32
    budgets: list              # [n_kept]
    sel: list                  # per kept tile, ascending dominant token indices
    ctx_targets: list = None   # per kept tile, the contextual tokens' targets (merge only)
    ctx_groups: list = None
    ctx: list = None           # per kept tile, fp64 [m, d] contextual tokens


def decide(r32, s32, G, m, policy, p_ext=None):
    """Every decision of a4-a7 from the fp32 scores and the fp64 similarities."""
    nbr = knn_neighbours(G, m)
    st = smooth(s32, nbr)
    u = minmax_normalize(st)
    kept = retained(u, policy.tau)
    if p_ext is None:
        p = np.array([u[i] for i in kept], dtype=F32)
    else:
        p = np.array([F32(p_ext[i]) for i in kept], dtype=F32)
    bud = [budget(float(pi), policy) for pi in p]
    n_v = r32.shape[1]
    sel = [top_b(r32[i], b - contextual_count(b, n_v, policy)) for i, b in zip(kept, bud)]
    return nbr, st, u, kept, p, bud, sel


def select(X, embed, query_ids, bg_ids, m, policy, p_ext=None, templates=None) -> Selection:
    t = query_embedding(embed, templates if templates is not None else [query_ids])
    B = background_embeddings(embed, bg_ids)
    r64, V, s64 = score_scene(X, t, B)
    r32, s32 = to_f32(r64), to_f32(s64)
    G = similarity(V)
    nbr, st, u, kept, p, bud, sel = decide(r32, s32, G, m, policy, p_ext)
    out = Selection(t, B, r64, V, s64, r32, s32, G, nbr, st, u, kept, p, bud, sel)
    if getattr(policy, "ctx_num", 0):
        n_v = X.shape[1]
        merged = [merge_contextual(X[i], idx, contextual_count(b, n_v, policy))
                  for i, idx, b in zip(kept, sel, bud)]
        out.ctx_targets = [mg[0] for mg in merged]
        out.ctx_groups = [mg[1] for mg in merged]
        out.ctx = [mg[2] for mg in merged]
    return out
