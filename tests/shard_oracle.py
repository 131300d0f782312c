"""The oracle as the per-rank engine of a sharded scene query (test infrastructure).

Each rank holds only its shard of tiles; every score and decision is the oracle's, taken from
what the protocol of paper_2609_29029_gb300.shard hands the rank (its own tiles, the gathered
tile embeddings and raw scores, the reduced score range).  Run over gloo ranks on the CPU, it
shows that the exchanges carry everything the scene-wide steps need: the union of the ranks'
results equals the oracle's single-rank selection.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import rift_oracle as O


class OracleShardEngine:
    def __init__(self, X_shard, embed, query_ids, bg_ids, sys_ids, knn_m, policy, get_layer=None, g_final=None,
                 dec=None):
        self.X, self.embed = X_shard, embed
        self.query_ids, self.bg_ids, self.sys_ids = query_ids, bg_ids, sys_ids
        self.knn_m, self.policy = knn_m, policy
        self.get_layer, self.g_final, self.dec = get_layer, g_final, dec

    def score_shard(self, lo, hi):
        assert self.X.shape[0] == hi - lo
        t = O.query_embedding(self.embed, [self.query_ids])
        B = O.background_embeddings(self.embed, self.bg_ids)
        r64, V, s64 = O.score_scene(self.X, t, B)
        self.r32 = O.to_f32(r64)
        return {"r": torch.from_numpy(self.r32), "s_raw": torch.from_numpy(O.to_f32(s64)), "V": V}

    def smooth_rows(self, V_all, s_all, lo, hi):
        nbr = O.knn_neighbours(O.similarity(V_all), self.knn_m)
        st = O.smooth(s_all.numpy(), nbr)
        return torch.from_numpy(st[lo:hi].copy()), torch.from_numpy(nbr[lo:hi].copy())

    def score_range(self, tile_s):
        s = tile_s.numpy()
        return torch.from_numpy(np.array([s.min(), s.max()], dtype=np.float32))

    def select(self, loc, tile_s, rng):
        u = O.minmax_normalize(tile_s.numpy(), lo=float(rng[0]), hi=float(rng[1]))
        kept = O.retained(u, self.policy.tau)
        bud = [O.budget(float(u[i]), self.policy) for i in kept]
        n_v = self.r32.shape[1]
        sel = [O.top_b(self.r32[i], b - O.contextual_count(b, n_v, self.policy)) for i, b in zip(kept, bud)]
        self._sel = (kept, bud, sel)
        return {"kept": kept, "budgets": bud, "sel": sel, "u": torch.from_numpy(u)}

    def pack(self, sel):
        kept, bud, idx = self._sel
        ctx = None
        if getattr(self.policy, "ctx_num", 0):
            n_v = self.X.shape[1]
            ctx = [O.merge_contextual(self.X[i], s, O.contextual_count(b, n_v, self.policy))[2]
                   for i, s, b in zip(kept, idx, bud)]
        H0, cu, pos = O.pack(self.X, self.embed, kept, idx, self.sys_ids, self.query_ids, ctx=ctx)
        return H0, cu, torch.tensor(pos, dtype=torch.int32)

    def prefill(self, rows, cu, positions):
        out = [O.prefill_sequence(rows[cu[j]:cu[j + 1]], self.get_layer, self.g_final, self.dec)
               for j in range(len(cu) - 1)]
        return torch.cat(out)
