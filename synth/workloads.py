"""The synthetic workloads: decoder shapes, budget policies and seeded scenes.

The paper measures on xView and GLH-Bridge scenes with RemoteCLIP embeddings
and trained LLaVA-1.5-7B weights (Section 3); none of those exist here.  These
seeded inputs stand in for them with the shapes the paper states: 336 px tiles
that each become 576 projected vision tokens (Section 1), scenes of 64 to
about 400 tiles (Section 1, Appendix B), a Vicuna-7B decoder shape, and a query
whose embedding rows point along a direction that is planted into a few
"relevant" tiles.

Nothing here computes a step of the method; it only makes inputs.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

from . import rng


@dataclass(frozen=True)
class DecoderShape:
    n_layers: int
    d: int
    n_heads: int
    head_dim: int
    ffn: int
    vocab: int
    eps: float = 1e-6
    rope_theta: float = 1e4

    @property
    def params_per_layer(self) -> int:
        return 4 * self.d * self.d + 3 * self.d * self.ffn

    @property
    def linear_flops_per_token(self) -> int:
        return 2 * self.n_layers * self.params_per_layer

    def attn_flops(self, L: int) -> int:
        """Causal attention FLOPs for one sequence of length L over all layers
        (QK^T and PV over the L(L+1)/2 unmasked pairs, 2 flop per MAC)."""
        return self.n_layers * 4 * self.n_heads * self.head_dim * (L * (L + 1) // 2)


LLAVA7B = DecoderShape(n_layers=32, d=4096, n_heads=32, head_dim=128, ffn=11008, vocab=32000)
TINY_DECODER = DecoderShape(n_layers=2, d=256, n_heads=4, head_dim=64, ffn=688, vocab=1000)


@dataclass(frozen=True)
class Policy:
    """Stage-1 threshold and the Stage-2 budget table of Eq. 2.

    C is ascending, so an argmax tie resolves to the lower index = the cheaper
    budget.  The alpha/energy values are synthetic (the paper gives them only in
    figures): alpha+ is flat in c and alpha- degrades under compression, which
    reproduces the walkthrough's "inverted" assignment (Appendix B, Step 4):
    confident tiles get 72 tokens, uncertain tiles 288.
    """
    tau: float
    C: tuple
    alpha_pos: tuple
    alpha_neg: tuple
    energy: tuple
    lam: float
    # Contextual tokens inside a budget c < n_v: floor(ctx_num c / ctx_den) of the c tokens are
    # merged from the unselected ones (Stage 2, VisionZip's mechanism); ctx_num = 0 selects only.
    ctx_num: int = 0
    ctx_den: int = 64


RIFT_POLICY = Policy(tau=0.37, C=(72, 144, 288, 432, 576),
                     alpha_pos=(0.86, 0.87, 0.875, 0.877, 0.878),
                     alpha_neg=(0.50, 0.68, 0.84, 0.868, 0.89),
                     energy=(0.28, 0.40, 0.62, 0.82, 1.00), lam=0.15)
RIFT_POLICY_SKEW = replace(RIFT_POLICY, lam=0.10)
# VisionZip's split of a budget into dominant and contextual tokens (54 + 10 of 64)
RIFT_POLICY_MERGE = replace(RIFT_POLICY, ctx_num=10, ctx_den=64)
# tau = 0 keeps every tile (u >= 0 always); C = {576} gives every tile its full budget.
KEEP_ALL = Policy(tau=0.0, C=(576,), alpha_pos=(1.0,), alpha_neg=(1.0,), energy=(0.0,), lam=0.0)


@dataclass(frozen=True)
class SceneSpec:
    N: int
    d: int
    x_dtype: str                 # "f32" or "bf16"
    n_v: int = 576
    grid: int = 24               # n_v = grid * grid token layout of one tile
    planted_frac: float = 0.05   # tiles carrying the query direction at full strength
    distractor_frac: float = 0.18  # "context" tiles: weak query direction + a background direction
    strength: str = "fixed"      # "fixed" or "pareto"
    alpha: float = 8.0           # planted amount per patch token along the unit query direction
    pareto_shape: float = 1.5
    M: int = 8                   # background vocabulary size
    S: int = 35                  # system-prompt tokens
    Q: int = 24                  # query tokens
    seed: int = 0


@dataclass(frozen=True)
class Workload:
    name: str
    scene: SceneSpec
    decoder: DecoderShape
    policy: Policy
    knn_m: int = 6
    description: str = ""

    @property
    def m_eff(self) -> int:
        return min(self.knn_m, self.scene.N - 1)


TINY = Workload(
    "tiny",
    SceneSpec(N=4, d=256, x_dtype="f32", planted_frac=0.25, distractor_frac=0.25, S=8, Q=16),
    TINY_DECODER, RIFT_POLICY, knn_m=6,
    description="4 tiles x 576 fp32 tokens (d=256), 2-layer hidden-256 decoder, prune + elastic budgets")
EXH16 = Workload(
    "exhaustive16_7b",
    SceneSpec(N=16, d=4096, x_dtype="bf16", planted_frac=0.10, distractor_frac=0.0),
    LLAVA7B, KEEP_ALL, knn_m=6,
    description="16 tiles x 576 bf16 tokens, 10% planted, keep-all full-budget prefill at the 7B shape")
EXH400 = Workload(
    "exhaustive400_7b",
    SceneSpec(N=400, d=4096, x_dtype="bf16"),
    LLAVA7B, KEEP_ALL, knn_m=6,
    description="400 tiles x 576 bf16 tokens, 5% planted + 12% distractors, keep-all prefill of 400 x 635 tokens")
RIFT400 = Workload(
    "rift400_7b",
    SceneSpec(N=400, d=4096, x_dtype="bf16"),
    LLAVA7B, RIFT_POLICY, knn_m=6,
    description="same 400-tile scene, tau=0.37 pruning, kNN-6 smoothing, elastic budgets, packed varlen prefill")
RIFT1600 = Workload(
    "rift1600_7b",
    SceneSpec(N=1600, d=4096, x_dtype="bf16", strength="pareto", distractor_frac=0.0, planted_frac=0.0),
    LLAVA7B, RIFT_POLICY_SKEW, knn_m=6,
    description="1600 tiles, Pareto(1.5) planted strengths on every tile, elastic budgets with lambda=0.10")

RIFT400_MERGE = replace(RIFT400, name="rift400_7b_merge", policy=RIFT_POLICY_MERGE,
                        description="the rift400_7b query with Stage 2's merge: each budget holds "
                                    "floor(10 c / 64) contextual tokens merged from the unselected ones")

WORKLOADS = {w.name: w for w in (TINY, EXH16, EXH400, RIFT400, RIFT1600, RIFT400_MERGE)}
SWEEP_N = (100, 400, 1600, 6400)


def sweep_workload(N: int) -> Workload:
    return replace(RIFT400, name=f"sweep{N}", scene=replace(RIFT400.scene, N=N))


# ----------------------------------------------------------------------------------------------
# Scene generation
# ----------------------------------------------------------------------------------------------

@dataclass
class Scene:
    spec: SceneSpec
    X: torch.Tensor              # [N, n_v, d] fp32 or bf16
    embed: torch.Tensor          # [vocab, d] bf16 (also the decoder's token embedding)
    sys_ids: list
    query_ids: list
    bg_ids: list
    planted: list                # tile indices with the full query direction
    distractors: list
    strength: list               # per-tile planted amount (host floats)
    patches: dict = field(default_factory=dict)  # tile -> list of token indices


def _tile_roles(spec: SceneSpec):
    n_p = int(round(spec.planted_frac * spec.N))
    n_d = int(round(spec.distractor_frac * spec.N))
    order = rng.permutation_prefix(spec.seed, rng.stream_id("roles"), spec.N, spec.N)
    planted = sorted(order[:n_p])
    distract = sorted(order[n_p:n_p + n_d])
    u = rng.uniform_f64_host(spec.seed, rng.stream_id("strength"), spec.N)
    strength = [0.0] * spec.N
    if spec.strength == "fixed":
        for i in planted:
            strength[i] = spec.alpha
        for i in distract:
            strength[i] = spec.alpha * (0.3 + 0.4 * u[i])
    elif spec.strength == "pareto":
        for i in range(spec.N):
            x = (1.0 - u[i]) ** (-1.0 / spec.pareto_shape) - 1.0
            strength[i] = spec.alpha * min(x, 64.0)
        planted = [i for i in range(spec.N) if strength[i] >= spec.alpha]
    else:
        raise ValueError(spec.strength)
    return planted, distract, strength


def _patch(spec: SceneSpec, i: int) -> list:
    u = rng.uniform_f64_host(spec.seed, rng.stream_id("patch", i), 4)
    h = 4 + int(u[0] * 5)
    w = 4 + int(u[1] * 5)
    r0 = int(u[2] * (spec.grid - h + 1))
    c0 = int(u[3] * (spec.grid - w + 1))
    return [(r0 + r) * spec.grid + (c0 + c) for r in range(h) for c in range(w)]


def make_scene(spec: SceneSpec, vocab: int, device="cpu", tile_block: int = 32) -> Scene:
    d = spec.d
    ids = rng.permutation_prefix(spec.seed, rng.stream_id("ids"), vocab, spec.S + spec.Q + spec.M)
    sys_ids, query_ids, bg_ids = ids[:spec.S], ids[spec.S:spec.S + spec.Q], ids[spec.S + spec.Q:]
    g = rng.sign_vector(spec.seed, rng.stream_id("query_dir"), d, device)
    h0 = rng.sign_vector(spec.seed, rng.stream_id("bg_dir", 0), d, device)

    planted, distract, strength = _tile_roles(spec)
    patches = {}
    for i in range(spec.N):
        if strength[i] > 0.0:
            patches[i] = _patch(spec, i)
    dset = set(distract)

    # Vision tokens: N(0,1) per element, plus (strength * g) on the patch tokens of planted
    # tiles; distractor ("context") tiles also get alpha * h0, a background direction.
    xdt = torch.float32 if spec.x_dtype == "f32" else torch.bfloat16
    X = torch.empty(spec.N, spec.n_v, d, dtype=xdt, device=device)
    per_tile = spec.n_v * d
    for b0 in range(0, spec.N, tile_block):
        b1 = min(spec.N, b0 + tile_block)
        blk = rng.normal_f32(spec.seed, rng.stream_id("X"), (b1 - b0) * per_tile, device,
                             offset=b0 * per_tile).view(b1 - b0, spec.n_v, d)
        for i in range(b0, b1):
            if i in patches:
                idx = torch.tensor(patches[i], dtype=torch.long, device=device)
                add = strength[i] * g
                if i in dset:
                    add = add + spec.alpha * h0
                blk[i - b0].index_add_(0, idx, add.expand(len(patches[i]), d).contiguous())
        X[b0:b1] = blk.to(xdt)

    # Embedding table N(0, 0.02); the query rows also carry beta * g and background row j
    # carries beta * h_j, beta = 0.02 * sqrt(d) (the norm of a noise row).
    beta = 0.02 * math.sqrt(d)
    E = rng.normal_f32(spec.seed, rng.stream_id("embed"), vocab * d, device).view(vocab, d) * 0.02
    qi = torch.tensor(query_ids, dtype=torch.long, device=device)
    E[qi] += beta * g
    for j, bid in enumerate(bg_ids):
        hj = h0 if j == 0 else rng.sign_vector(spec.seed, rng.stream_id("bg_dir", j), d, device)
        E[bid] += beta * hj
    embed = E.to(torch.bfloat16)
    return Scene(spec, X, embed, sys_ids, query_ids, bg_ids, planted, distract, strength, patches)


# ----------------------------------------------------------------------------------------------
# Decoder weights (random init N(0, 0.02), bf16; norm gains 1 + 0.1 N(0,1) so that a wrong
# gain index is visible in tests).  Logical layout: [out_features, in_features].
# ----------------------------------------------------------------------------------------------

LAYER_TENSORS = ("wq", "wk", "wv", "wo", "wg", "wu", "wd", "g_attn", "g_ffn")


def layer_shapes(dec: DecoderShape) -> dict:
    d, f = dec.d, dec.ffn
    return {"wq": (d, d), "wk": (d, d), "wv": (d, d), "wo": (d, d),
            "wg": (f, d), "wu": (f, d), "wd": (d, f), "g_attn": (d,), "g_ffn": (d,)}


def _weight(seed: int, name: str, layer: int, shape, device) -> torch.Tensor:
    n = 1
    for s in shape:
        n *= s
    z = rng.normal_f32(seed, rng.stream_id("w", layer, name), n, device).view(*shape)
    if name.startswith("g_"):
        return (1.0 + 0.1 * z).to(torch.bfloat16)
    return (z * 0.02).to(torch.bfloat16)


def make_layer(dec: DecoderShape, layer: int, device="cpu", seed: int = 0) -> dict:
    return {k: _weight(seed, k, layer, s, device) for k, s in layer_shapes(dec).items()}


def make_final_norm(dec: DecoderShape, device="cpu", seed: int = 0) -> torch.Tensor:
    return _weight(seed, "g_final", -1, (dec.d,), device)


def make_lm_head(dec: DecoderShape, device="cpu", seed: int = 0) -> torch.Tensor:
    """Untied output matrix [vocab, d] (LLaMA/Vicuna keep it separate from the embedding)."""
    return _weight(seed, "lm_head", -1, (dec.vocab, dec.d), device)
