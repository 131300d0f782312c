"""Shared helpers of the GPU parity tests: workloads at test sizes, running the CUDA path
through the C ABI, running the oracle, and the decision-margin checks.

Decisions are integers decided by fp32 values.  The oracle rounds fp64 scores once to fp32;
the CUDA path accumulates in fp32 in another order, so its fp32 scores differ in the last
bits.  Where the oracle's own margin of a decision exceeds the bound on that difference, the
decision is unique and both sides must agree exactly; the test inputs are seeded so that every
decision clears its bound (``margins`` reports any that do not, and the tests assert none).
"""
from __future__ import annotations

from dataclasses import replace

import numpy as np
import torch

from oracle import rift_oracle as O
from synth import workloads as W

F32 = np.float32

# Bounds on |CUDA fp32 - oracle fp32| of the quantities that decide integers (score-relative).
SCORE_RTOL = 1e-4    # token and tile scores, relative to the largest magnitude of their row/scene
HIDDEN_TOL = 2e-2    # final hidden states, max |g - o| / max |o| per sequence

# Small extra workloads: several tiles, pruning, ragged tails, both input dtypes.
SMALL24 = W.Workload("small24_f32", W.SceneSpec(N=24, d=256, x_dtype="f32", planted_frac=0.1,
                                                distractor_frac=0.15, S=8, Q=16),
                     W.TINY_DECODER, W.RIFT_POLICY, knn_m=6)
# n_v = 200: the budget set C scaled from {72, ..., 576} of 576 tokens to 200 tokens
RAGGED = W.Workload("ragged40_bf16", W.SceneSpec(N=40, d=256, x_dtype="bf16", n_v=200, grid=14,
                                                 planted_frac=0.1, distractor_frac=0.2, S=5, Q=7, M=3),
                    W.TINY_DECODER, replace(W.RIFT_POLICY_SKEW, C=(25, 50, 100, 150, 200)), knn_m=4)


def to_dev(sc, device):
    i32 = dict(dtype=torch.int32, device=device)
    return dict(X=sc.X.to(device), embed=sc.embed.to(device),
                q=torch.tensor(sc.query_ids, **i32), bg=torch.tensor(sc.bg_ids or [0], **i32),
                sys=torch.tensor(sc.sys_ids or [0], **i32))


def gpu_pipeline(wl, sc, device, model=None, p=None, max_T=None):
    from paper_2609_29029_gb300 import ScenePipeline
    s = wl.scene
    pipe = ScenePipeline(s.N, s.n_v, s.d, s.x_dtype, s.M, s.S, s.Q, wl.knn_m, wl.policy, model=model,
                         max_T=max_T, device=device)
    return pipe, to_dev(sc, device)


def oracle_select(wl, sc, p_ext=None):
    return O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy, p_ext=p_ext)


class HostTiles:
    """A device scene X [N, n_v, d] handed to the oracle tile by tile: indexing copies a block of
    tiles to the host, so a scene larger than host memory (30 GB at 6400 tiles) never has to be
    copied whole.  The values are the generator's, unchanged."""

    def __init__(self, X, block: int = 64):
        self.X, self.block = X, block
        self.shape = tuple(X.shape)
        self._b0, self._blk = -1, None

    def __len__(self):
        return self.shape[0]

    def __getitem__(self, i):
        i = int(i)
        b0 = (i // self.block) * self.block
        if b0 != self._b0:
            self._blk = self.X[b0:b0 + self.block].cpu()
            self._b0 = b0
        return self._blk[i - b0]


# Bounds on |CUDA fp32 value - oracle fp32 value| of the quantities that decide integers.
#  * similarity G (compared in fp64 on both sides): the CUDA path recomputes its kNN candidates
#    with fp64 accumulation of the fp32 tile embeddings, whose elements carry ~1e-7 relative error
#    from the fp32 pooled sums; in a 4096-term dot product that averages to ~3e-9; bound 3e-8.
#  * tile score, utility: fp32 dot products whose running sums cancel: ~1e-7; bounds 1e-6.
#  * token score r = x.w / ||x||: ~5e-9 absolute; bound 2e-6 of the tile's largest |r|.
EPS_G = 3e-8        # cosine similarity of two tiles (|G| <= 1)
EPS_S = 1e-6        # tile score, relative to max |s~| over the scene
EPS_U = 1e-6        # utility U(c) (|dU/dp| <= 0.4, p = u)
EPS_R = 2e-6        # token score, relative to max |r| over the tile

# Seeds whose scene has every kNN / threshold / budget decision clear of its bound.  Seed 0 of the
# 1600-tile scene has a kNN gap of 1.3e-8 and a kept tile whose p = 0.8903232 is one of the 11
# fp32 values in [0.37, 1] where two utilities of the lambda = 0.10 table are equal; seed 3 clears
# every bound (its remaining top-b near-ties are checked for validity).
PARITY_SEED = {"rift1600_7b": 3}


def parity_workload(wl):
    seed = PARITY_SEED.get(wl.name, wl.scene.seed)
    return replace(wl, scene=replace(wl.scene, seed=seed))


def margins(sel: O.Selection, wl) -> dict:
    """The oracle's smallest margin of each kind of decision, in units of its bound (>= 1: the
    decision is unique at the precision the CUDA path reaches).  'topb_tiles' lists the kept
    slots whose rank-b gap is below its bound."""
    out = {}
    N = len(sel.s32)
    m = min(wl.knn_m, N - 1)
    worst = np.inf
    if 0 < m < N - 1:
        for i in range(N):
            g = np.sort(np.delete(sel.G[i].astype(np.float64), i))[::-1]
            worst = min(worst, (g[m - 1] - g[m]) / EPS_G)
    out["knn"] = worst
    st = sel.s_tilde.astype(np.float64)
    span = st.max() - st.min()
    if wl.policy.tau <= 0.0:
        out["tau"] = np.inf  # u >= 0 holds exactly (s~ - min >= 0), so nothing can flip
    elif span > 0:
        du = 3 * EPS_S * np.abs(st).max() / span
        out["tau"] = float(np.min(np.abs(sel.u.astype(np.float64) - float(F32(wl.policy.tau)))) / du)
    else:
        out["tau"] = np.inf
    wb = np.inf
    for p in sel.p:
        U = sorted([float(x) for x in O.utility(float(p), wl.policy)], reverse=True)
        if len(U) > 1:
            wb = min(wb, (U[0] - U[1]) / EPS_U)
    out["budget"] = wb
    wt, amb = np.inf, []
    for j, (i, idx) in enumerate(zip(sel.kept, sel.sel)):
        b = len(idx)  # the selected tokens: the budget less its contextual tokens when merging
        r = np.sort(sel.r32[i].astype(np.float64))[::-1]
        if 0 < b < len(r):
            mj = (r[b - 1] - r[b]) / (EPS_R * np.abs(r).max())
            wt = min(wt, mj)
            if mj < 1.0:
                amb.append(j)
    out["topb"] = wt
    out["topb_tiles"] = amb
    return out


def assert_margins(sel, wl, allow_topb=False):
    """Every kNN, threshold and budget decision must clear its bound; top-b decisions too unless
    allow_topb (then the ambiguous slots are returned and checked for validity instead)."""
    mg = margins(sel, wl)
    keys = ["knn", "tau", "budget"] + ([] if allow_topb else ["topb"])
    bad = {k: mg[k] for k in keys if not mg[k] >= 1.0}
    assert not bad, f"seeded input has decisions closer than the fp32 bound: {bad}"
    return set(mg["topb_tiles"])


def topb_is_valid(gpu_idx, r32_tile, b):
    """A selection that differs from the oracle's only inside the fp32 bound of the boundary:
    b indices, ascending, every token clearly above the b-th score taken, none clearly below."""
    r = np.asarray(r32_tile, dtype=np.float64)
    if len(gpu_idx) != b or list(gpu_idx) != sorted(set(gpu_idx)):
        return False
    vb = np.sort(r)[::-1][b - 1]
    eps = EPS_R * np.abs(r).max()
    chosen = set(gpu_idx)
    must = {k for k in range(len(r)) if r[k] > vb + eps}
    never = {k for k in range(len(r)) if r[k] < vb - eps}
    return must <= chosen and not (chosen & never)


def neighbours_match(gpu_nbr, sel) -> list:
    """Rows whose neighbour SET differs from the oracle's (the set is what the smoothing uses),
    plus rows whose emitted rank order contradicts the oracle's similarities by more than the
    bound.  Equal sets with a swapped near-tie (|dG| < EPS_G) are accepted."""
    bad = []
    for i in range(len(gpu_nbr)):
        g = [int(j) for j in gpu_nbr[i]]
        if sorted(g) != sorted(int(j) for j in sel.nbr[i]):
            bad.append(i)
            continue
        if any(sel.G[i, g[k]] < sel.G[i, g[k + 1]] - EPS_G for k in range(len(g) - 1)):
            bad.append(i)
    return bad


def rel_err_rows(g: np.ndarray, o: np.ndarray) -> float:
    """max |g - o| / max |o| over each row, maximised over rows."""
    g = np.atleast_2d(g).astype(np.float64)
    o = np.atleast_2d(o).astype(np.float64)
    den = np.maximum(np.abs(o).max(axis=1), 1e-30)
    return float((np.abs(g - o).max(axis=1) / den).max())


def max_abs_rel(g, o) -> float:
    g = torch.as_tensor(g).double()
    o = torch.as_tensor(o).double()
    return float((g - o).abs().max() / o.abs().max().clamp_min(1e-30))


def seq_slices(cu):
    return [(int(cu[j]), int(cu[j + 1])) for j in range(len(cu) - 1)]


def with_policy(wl, policy):
    return replace(wl, policy=policy)
