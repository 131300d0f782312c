"""One scene query sharded over R ranks.

Every step of Rift is per tile except two that need the whole scene: the kNN smoothing of
Appendix B Step 2 (a tile's m most similar tiles may sit in any shard) and the per-scene min-max
of Section 2.3 Stage 1.  So a scene split into contiguous shards of tiles needs exactly two
exchanges before its selection, plus one to balance the prefill:

  1. each rank scores its shard (Eq. 1 on tokens and tiles) and forms its tile embeddings V;
  2. exchange: all-gather of V and of the raw tile scores (tile order = rank order);
  3. each rank smooths its own tiles against the whole scene;
  4. exchange: all-reduce of (min, max) of the smoothed scores;
  5. each rank prunes, budgets and selects the tokens of its own tiles with the scene's range,
     and packs its kept tiles' sequences;
  6. exchange: all-gather of every kept tile's (tile id, sequence length); every rank computes the
     same cost-balanced assignment of sequences to ranks, and an all-to-all moves each packed
     sequence from the rank that owns its tile to the rank that prefills it;
  7. each rank prefills its sequences (weights replicated).

The protocol is written once, as a generator per rank that yields its exchange requests
(Gather, MinMax, AllToAll).  run_group() serves them with torch.distributed collectives over a
process group (gloo on CPU tensors, NCCL on GPU tensors); run_inprocess() serves the generators of
all ranks of one process in lockstep (several ranks' shards on one device, the exchanges done by
concatenation).  Elastic membership (a rank that leaves between queries) is Membership below.

The per-rank compute is an engine object; CudaShardEngine runs every step through the C ABI of
libriftgb.so.  The library itself makes no collective call.
"""
from __future__ import annotations

import time
from dataclasses import dataclass, field

import torch

from . import abi


# ------------------------------------------------------------------------------- exchange requests

@dataclass
class Gather:
    """All-gather along dim 0 (shards may differ in size); the result is the concatenation in
    rank order."""
    tensor: torch.Tensor


@dataclass
class MinMax:
    """All-reduce of a (min, max) pair: the min of the mins and the max of the maxes."""
    tensor: torch.Tensor


@dataclass
class AllToAll:
    """tensors[q] goes to rank q (dim 0 may differ); the result lists what came from each rank."""
    tensors: list


# ------------------------------------------------------------------------------- sharding

def shard_bounds(N: int, R: int) -> list:
    """Contiguous shards: rank r holds tiles bounds[r] .. bounds[r + 1] - 1 (sizes differ by at
    most one)."""
    if N < R:
        raise ValueError(f"{N} tiles cannot be split over {R} ranks")
    return [(N * r) // R for r in range(R + 1)]


def sequence_cost(L: int, dec) -> int:
    """FLOPs of prefilling one sequence of L rows: the linear layers per row plus causal attention."""
    return L * dec.linear_flops_per_token + dec.attn_flops(L)


def rebalance(seqs: list, R: int, dec) -> list:
    """Assignment of sequences [(tile id, L)] to R ranks: longest processing time first (by
    decreasing cost, ties to the lower tile id), each to the rank with the least cost so far (ties
    to the lower rank).  Returns the tile ids of each rank, ascending.  Every rank computes the
    same assignment from the same gathered list."""
    load = [0] * R
    out = [[] for _ in range(R)]
    for tile, L in sorted(seqs, key=lambda s: (-sequence_cost(s[1], dec), s[0])):
        q = min(range(R), key=lambda r: (load[r], r))
        load[q] += sequence_cost(L, dec)
        out[q].append(tile)
    return [sorted(o) for o in out]


@dataclass
class ShardResult:
    """What one rank holds after a sharded query."""
    bounds: list                  # the tile shards of all ranks
    kept: list                    # global ids of this rank's kept tiles (the ones it selected)
    budgets: list                 # b_j of each, in that order
    sel: list                     # selected token indices of each (ascending)
    u: torch.Tensor               # u of this rank's shard
    nbr: torch.Tensor             # NN of this rank's tiles (global tile ids)
    tile_s: torch.Tensor          # smoothed scores of this rank's tiles
    seq_tiles: list = field(default_factory=list)   # tiles whose sequences this rank prefilled
    rows: torch.Tensor = None     # their packed rows [T, d] (after the prefill: final hidden states)
    cu: list = None               # their offsets


def sharded_query(engine, rank: int, R: int, N: int, dec=None, prefill: bool = True):
    """The protocol of one rank (a generator: it yields exchange requests and receives their
    results).  engine: the per-rank compute (see CudaShardEngine)."""
    bounds = shard_bounds(N, R)
    lo, hi = bounds[rank], bounds[rank + 1]
    loc = engine.score_shard(lo, hi)
    # 2. the scene's tile embeddings and raw scores
    V_all = yield Gather(loc["V"])
    s_all = yield Gather(loc["s_raw"])
    # 3. this shard's smoothing against the whole scene
    tile_s, nbr = engine.smooth_rows(V_all, s_all, lo, hi)
    # 4. the scene's range of smoothed scores
    rng = yield MinMax(engine.score_range(tile_s))
    # 5. prune, budgets, top-b and packing of this shard's tiles
    sel = engine.select(loc, tile_s, rng)
    kept = [lo + j for j in sel["kept"]]
    packed, cu, pos = engine.pack(sel)
    res = ShardResult(bounds, kept, sel["budgets"], sel["sel"], sel["u"], nbr, tile_s)
    # 6. balance the prefill: every kept sequence's (tile, length), then the rows to their rank
    meta = torch.tensor([[t, cu[j + 1] - cu[j]] for j, t in enumerate(kept)], dtype=torch.int64,
                        device=packed.device).reshape(-1, 2)
    meta_all = yield Gather(meta)
    seqs = [(int(t), int(L)) for t, L in meta_all.tolist()]
    assign = rebalance(seqs, R, dec) if dec is not None else [[t for t, _ in seqs if bounds[q] <= t < bounds[q + 1]]
                                                               for q in range(R)]
    owner_row = {t: j for j, t in enumerate(kept)}
    send_rows, send_pos = [], []
    for q in range(R):
        mine = [owner_row[t] for t in assign[q] if t in owner_row]
        send_rows.append(torch.cat([packed[cu[j]:cu[j + 1]] for j in mine]) if mine else packed[:0])
        send_pos.append(torch.cat([pos[cu[j]:cu[j + 1]] for j in mine]) if mine else pos[:0])
    got_rows = yield AllToAll(send_rows)
    got_pos = yield AllToAll(send_pos)
    # the sequences arrive by owner rank, each owner's in ascending tile order: ascending overall
    res.seq_tiles = assign[rank]
    lengths = dict(seqs)
    res.cu = [0]
    for t in res.seq_tiles:
        res.cu.append(res.cu[-1] + lengths[t])
    res.rows = torch.cat(got_rows) if got_rows else packed[:0]
    positions = torch.cat(got_pos) if got_pos else pos[:0]
    assert res.rows.shape[0] == res.cu[-1]
    # 7. prefill this rank's sequences
    if prefill and dec is not None and res.seq_tiles:
        res.rows = engine.prefill(res.rows, res.cu, positions)
    return res


# ------------------------------------------------------------------------------- drivers

def _collective(req, group):
    """Serve one exchange request with torch.distributed over `group` (tensors stay where they
    are: CPU tensors for gloo, CUDA tensors for NCCL)."""
    import torch.distributed as dist
    R = dist.get_world_size(group)
    if isinstance(req, MinMax):
        t = req.tensor
        both = torch.stack([t[0], -t[1]])  # negation is exact: one MIN reduction serves both
        dist.all_reduce(both, op=dist.ReduceOp.MIN, group=group)
        return torch.stack([both[0], -both[1]])
    if isinstance(req, Gather):
        t = req.tensor.contiguous()
        n = torch.tensor([t.shape[0]], dtype=torch.int64, device=t.device)
        sizes = [torch.zeros_like(n) for _ in range(R)]
        dist.all_gather(sizes, n, group=group)
        sizes = [int(s.item()) for s in sizes]
        pad = max(sizes)
        buf = torch.zeros((pad,) + tuple(t.shape[1:]), dtype=t.dtype, device=t.device)
        buf[:t.shape[0]] = t
        parts = [torch.empty_like(buf) for _ in range(R)]
        dist.all_gather(parts, buf, group=group)
        return torch.cat([p[:s] for p, s in zip(parts, sizes)])
    if isinstance(req, AllToAll):
        # 16-bit floats travel as their bytes (every backend moves uint8)
        dt0 = req.tensors[0].dtype
        as_bits = dt0 in (torch.bfloat16, torch.float16)
        ts = [(t.contiguous().view(torch.uint8) if as_bits else t.contiguous()) for t in req.tensors]
        dev, dt, tail = ts[0].device, ts[0].dtype, tuple(ts[0].shape[1:])
        row = 1
        for x in tail:
            row *= x
        n_out = torch.tensor([t.shape[0] for t in ts], dtype=torch.int64, device=dev)
        n_in = torch.empty_like(n_out)
        dist.all_to_all_single(n_in, n_out, group=group)
        n_in = [int(x) for x in n_in.tolist()]
        flat_out = torch.cat([t.reshape(-1) for t in ts])
        flat_in = torch.empty(sum(n_in) * row, dtype=dt, device=dev)
        dist.all_to_all_single(flat_in, flat_out, [c * row for c in n_in], [t.shape[0] * row for t in ts],
                               group=group)
        out, o = [], 0
        for c in n_in:
            part = flat_in[o:o + c * row].reshape((c,) + tail)
            out.append(part.view(dt0) if as_bits else part)
            o += c * row
        return out
    raise TypeError(f"unknown exchange request {req!r}")


def run_group(protocol, group=None):
    """Drive one rank's protocol generator over a torch.distributed process group."""
    try:
        req = next(protocol)
        while True:
            req = protocol.send(_collective(req, group))
    except StopIteration as e:
        return e.value


def run_inprocess(protocols: list) -> list:
    """Drive the protocols of all R ranks of one process in lockstep: at each exchange every rank
    has posted the same kind of request, served by concatenation (no collective library)."""
    R = len(protocols)
    reqs = [next(p) for p in protocols]
    done = [None] * R
    while True:
        kinds = {type(r) for r in reqs if r is not None}
        if not kinds:
            return done
        if len(kinds) != 1 or any(r is None for r in reqs):
            raise RuntimeError(f"ranks out of step: {[type(r).__name__ for r in reqs]}")
        if isinstance(reqs[0], Gather):
            cat = torch.cat([r.tensor for r in reqs])
            res = [cat] * R
        elif isinstance(reqs[0], MinMax):
            lo = torch.stack([r.tensor[0] for r in reqs]).min()
            hi = torch.stack([r.tensor[1] for r in reqs]).max()
            res = [torch.stack([lo, hi])] * R
        else:
            res = [[reqs[src].tensors[q] for src in range(R)] for q in range(R)]
        for r, p in enumerate(protocols):
            try:
                reqs[r] = p.send(res[r])
            except StopIteration as e:
                reqs[r], done[r] = None, e.value


class Membership:
    """Which ranks take part in a query, through a torch.distributed Store (the one the process
    group was made with).  Before query `step` every live rank announces itself; a rank that
    leaves says so (leave()), and a rank that neither announces itself nor leaves within
    `timeout` seconds is counted as gone.  Every survivor sees the same list, forms a process
    group of the survivors (new_group with local synchronization: the departed ranks take no part)
    and re-shards the scene over it."""

    def __init__(self, store, rank: int, world: int, timeout: float = 30.0):
        self.store, self.rank, self.world, self.timeout = store, rank, world, timeout

    def leave(self):
        self.store.set(f"rift_left/{self.rank}", "1")

    def live(self, step: int) -> list:
        self.store.set(f"rift_alive/{step}/{self.rank}", "1")
        t0 = time.monotonic()
        pending = set(range(self.world)) - {self.rank}
        alive = {self.rank}
        while pending:
            for r in sorted(pending):
                if self.store.check([f"rift_alive/{step}/{r}"]):
                    alive.add(r)
                    pending.discard(r)
                elif self.store.check([f"rift_left/{r}"]):
                    pending.discard(r)
            if pending and time.monotonic() - t0 > self.timeout:
                break
            if pending:
                time.sleep(0.01)
        return sorted(alive)

    def group(self, step: int):
        """(process group of the live ranks, this rank's index in it, their count)."""
        import torch.distributed as dist
        live = self.live(step)
        if len(live) == self.world:
            return None, self.rank, self.world
        g = dist.new_group(live, use_local_synchronization=True)
        return g, live.index(self.rank), len(live)


# ------------------------------------------------------------------------------- the CUDA engine

class CudaShardEngine:
    """One rank's compute of a sharded query through libriftgb.so.

    X_shard: the rank's tiles [hi - lo, n_v, d] (bf16 or fp32) on its GPU; the query (embed, ids)
    and, for the prefill, a DeviceModel are replicated.  Every score and decision is a kernel;
    host code only moves sizes and rows for the exchanges."""

    def __init__(self, X_shard, embed, phrase_ids, bg_ids, sys_ids, query_ids, M, S, Q, knn_m, policy,
                 model=None, stream=None):
        self.X = X_shard
        self.embed, self.phrase_ids, self.bg_ids = embed, phrase_ids, bg_ids
        self.sys_ids, self.query_ids = sys_ids, query_ids
        self.n_v, self.d = X_shard.shape[1], X_shard.shape[2]
        self.xdt = abi.RIFT_BF16 if X_shard.dtype == torch.bfloat16 else abi.RIFT_F32
        self.M, self.S, self.Q, self.knn_m = M, S, Q, knn_m
        self.policy = abi.make_policy(policy)
        num, den = getattr(policy, "ctx_num", 0), getattr(policy, "ctx_den", 64)
        self.max_m = max([(num * c) // den for c in policy.C if c < self.n_v] + [0]) if num else 0
        self.model = model
        self.stream = stream
        self.dev = X_shard.device

    def _f32(self, *shape):
        return torch.empty(*shape, dtype=torch.float32, device=self.dev)

    def _i32(self, *shape):
        return torch.empty(*shape, dtype=torch.int32, device=self.dev)

    def score_shard(self, lo, hi):
        n, d, st = hi - lo, self.d, self.stream
        t, B = self._f32(d), self._f32(max(self.M, 1), d)
        abi.query_prep(self.embed, self.embed.shape[0], d, self.phrase_ids, 1, self.phrase_ids.numel(),
                       self.bg_ids if self.M else None, self.M, t, B if self.M else None, st)
        r, s_raw, V = self._f32(n, self.n_v), self._f32(n), self._f32(n, d)
        need = abi.score_shard_workspace_bytes(n, self.n_v, d)
        ws = torch.empty(need, dtype=torch.uint8, device=self.dev)
        abi.score_shard(self.X, self.xdt, n, self.n_v, d, t, B if self.M else None, self.M, r, s_raw, V, ws, need, st)
        self.t, self.B, self.n = t, B, n
        return {"r": r, "s_raw": s_raw, "V": V}

    def smooth_rows(self, V_all, s_all, lo, hi):
        N, n = V_all.shape[0], hi - lo
        m = min(self.knn_m, N - 1)
        tile_s, nbr = self._f32(n), self._i32(max(n * m, 1))
        need = abi.smooth_workspace_bytes(N, n, self.d)
        ws = torch.empty(need, dtype=torch.uint8, device=self.dev)
        abi.smooth_rows(V_all.contiguous(), s_all.contiguous(), N, self.d, lo, n, self.knn_m, tile_s,
                        nbr if m > 0 else None, ws, need, self.stream)
        return tile_s, nbr[:n * m].view(n, m)

    def score_range(self, tile_s):
        rng = self._f32(2)
        abi.score_range(tile_s, tile_s.numel(), rng, self.stream)
        return rng

    def select(self, loc, tile_s, rng):
        n, n_v = self.n, self.n_v
        u, kept, n_kept = self._f32(n), self._i32(n), self._i32(1)
        budgets, sel, sel_off = self._i32(n), self._i32(n * n_v), self._i32(n + 1)
        abi.select_budgeted_tokens_ranged(loc["r"], tile_s, n, n_v, rng.to(self.dev), None, self.policy, u, kept,
                                          n_kept, budgets, sel, sel_off, self.stream)
        abi.sync_status(self.stream)
        k = int(n_kept.item())
        off = sel_off[:k + 1].tolist()
        s_all = sel.tolist()
        self._sel = (kept, n_kept, budgets, sel, sel_off)
        return {"kept": kept[:k].tolist(), "budgets": budgets[:k].tolist(),
                "sel": [s_all[off[j]:off[j + 1]] for j in range(k)], "u": u}

    def pack(self, sel):
        """The shard's kept tiles packed as [system | tokens (| contextual) | query] sequences:
        (rows bf16 [T, d], host offsets, positions int32 [T])."""
        kept, n_kept, budgets, sel_t, sel_off = self._sel
        n, n_v, d, st = self.n, self.n_v, self.d, self.stream
        ctx = ctx_off = None
        if self.max_m:
            max_ctx = n * self.max_m
            ctx = torch.empty(max(max_ctx, 1), d, dtype=torch.bfloat16, device=self.dev)
            ctx_off, ctx_t = self._i32(n + 1), self._i32(max(max_ctx, 1))
            need = abi.merge_workspace_bytes(n, n_v)
            ws = torch.empty(need, dtype=torch.uint8, device=self.dev)
            abi.merge_contextual(self.X, self.xdt, n, n_v, d, kept, n_kept, budgets, sel_t, sel_off, ctx, max_ctx,
                                 ctx_off, ctx_t, ws, need, st)
        k = len(sel["kept"])
        max_T = max(sum(self.S + b + self.Q for b in sel["budgets"]), 1)
        packed = torch.empty(max_T, d, dtype=torch.bfloat16, device=self.dev)
        cu, pos, T = self._i32(n + 1), self._i32(max_T), self._i32(1)
        abi.pack_ragged(self.X, self.xdt, n, n_v, d, kept, n_kept, sel_t, sel_off, self.sys_ids if self.S else None,
                        self.S, self.query_ids, self.Q, self.embed, self.embed.shape[0], packed, max_T, cu, pos, T, st,
                        ctx=ctx, ctx_off=ctx_off)
        abi.sync_status(st)
        Tn = int(T.item())
        return packed[:Tn], cu[:k + 1].tolist(), pos[:Tn]

    def prefill(self, rows, cu, positions):
        T, n_seq = rows.shape[0], len(cu) - 1
        max_len = max(cu[j + 1] - cu[j] for j in range(n_seq))
        hid = rows.contiguous().clone()
        cu_d = torch.tensor(cu, dtype=torch.int32, device=self.dev)
        need = abi.prefill_workspace_bytes(self.model.struct, T, n_seq, max_len)
        ws = torch.empty(need, dtype=torch.uint8, device=self.dev)
        abi.prefill_layers(self.model.struct, hid, T, cu_d, n_seq, max_len, positions.contiguous(), ws, need,
                           self.stream)
        abi.sync_status(self.stream)
        return hid
