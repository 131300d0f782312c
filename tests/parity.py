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


DECISION_EPS = 1e-5  # relative bound on the fp32 score difference that a decision must clear


def margins(sel: O.Selection, wl) -> dict:
    """The oracle's smallest margin of each kind of decision, in units of the bound on the
    CUDA/oracle score difference (>= 1 means the decision is unique at fp32 precision)."""
    out = {}
    N = len(sel.s32)
    m = min(wl.knn_m, N - 1)
    worst = np.inf
    if 0 < m < N - 1:
        for i in range(N):
            g = np.sort(np.delete(sel.G32[i].astype(np.float64), i))[::-1]
            worst = min(worst, (g[m - 1] - g[m]) / DECISION_EPS)
    out["knn"] = worst
    st = sel.s_tilde.astype(np.float64)
    span = st.max() - st.min()
    if span > 0:
        du = 3 * DECISION_EPS * np.abs(st).max() / span
        out["tau"] = float(np.min(np.abs(sel.u.astype(np.float64) - float(F32(wl.policy.tau)))) / du)
    else:
        out["tau"] = np.inf
    wb = np.inf
    for p in sel.p:
        U = sorted([float(x) for x in O.utility(float(p), wl.policy)], reverse=True)
        if len(U) > 1:
            wb = min(wb, (U[0] - U[1]) / DECISION_EPS)
    out["budget"] = wb
    wt = np.inf
    for i, b in zip(sel.kept, sel.budgets):
        r = np.sort(sel.r32[i].astype(np.float64))[::-1]
        if b < len(r):
            wt = min(wt, (r[b - 1] - r[b]) / (DECISION_EPS * np.abs(r).max()))
    out["topb"] = wt
    return out


def assert_margins(sel, wl):
    mg = margins(sel, wl)
    bad = {k: v for k, v in mg.items() if not v >= 1.0}
    assert not bad, f"seeded input has decisions closer than the fp32 bound: {bad}"


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
