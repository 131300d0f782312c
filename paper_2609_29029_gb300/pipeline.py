"""Device buffers and the call sequence of one scene query through the C ABI.

This module owns memory (torch tensors) and issues the five ABI calls in order; every
computation is a kernel of libriftgb.so.  The prefill reads the counts the selection and the
packing leave on the device (n_kept, T), so a whole query is enqueued without waiting for the
GPU; the counts are read back only for reporting (read_counts).
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

import torch

from . import abi


def interleave_gate_up(wg: torch.Tensor, wu: torch.Tensor) -> torch.Tensor:
    """[2F, d] with W_gate and W_up interleaved in 16-row groups (the layout rift_model wants)."""
    F, d = wg.shape
    assert F % 16 == 0 and wu.shape == wg.shape
    return torch.stack([wg.view(F // 16, 16, d), wu.view(F // 16, 16, d)], dim=1).reshape(2 * F, d).contiguous()


class DeviceModel:
    """Decoder weights in the library's layout plus the rift_model struct that points at them.

    Projection weights are stored in fp16 (the GEMM operand type; bf16 weights convert exactly
    unless their magnitude is below 2^-14, where fp16 keeps 2^-24 absolute resolution).  Norm
    gains stay bf16."""

    def __init__(self, dec, layers: list, g_final: torch.Tensor, device="cuda", lm_head: torch.Tensor | None = None):
        self.dec = dec
        self.layers = []
        h = torch.float16
        for W in layers:
            self.layers.append({
                "qkv": torch.cat([W["wq"], W["wk"], W["wv"]], 0).to(device).to(h).contiguous(),
                "o": W["wo"].to(device).to(h).contiguous(),
                "gate_up": interleave_gate_up(W["wg"].to(device), W["wu"].to(device)).to(h),
                "down": W["wd"].to(device).to(h).contiguous(),
                "g_attn": W["g_attn"].to(device, torch.bfloat16).contiguous(),
                "g_ffn": W["g_ffn"].to(device, torch.bfloat16).contiguous(),
            })
        self.g_final = g_final.to(device, torch.bfloat16).contiguous()
        n = len(self.layers)
        arr = C.c_void_p * n
        self._ptrs = {k: arr(*[L[k].data_ptr() for L in self.layers])
                      for k in ("qkv", "o", "gate_up", "down", "g_attn", "g_ffn")}
        m = abi.Model()
        m.n_layers, m.d, m.n_heads, m.head_dim, m.ffn = n, dec.d, dec.n_heads, dec.head_dim, dec.ffn
        m.eps, m.rope_theta = dec.eps, dec.rope_theta
        m.w_qkv, m.w_o = self._ptrs["qkv"], self._ptrs["o"]
        m.w_gate_up, m.w_down = self._ptrs["gate_up"], self._ptrs["down"]
        m.g_attn, m.g_ffn = self._ptrs["g_attn"], self._ptrs["g_ffn"]
        m.g_final = self.g_final.data_ptr()
        self.lm_head = None if lm_head is None else lm_head.to(device).to(h).contiguous()
        m.vocab = 0 if lm_head is None else lm_head.shape[0]
        m.lm_head = None if lm_head is None else self.lm_head.data_ptr()
        self.struct = m


@dataclass
class QueryResult:
    n_kept: int
    T: int
    t: torch.Tensor
    token_scores: torch.Tensor
    tile_s_raw: torch.Tensor
    tile_s: torch.Tensor
    nbr: torch.Tensor
    u: torch.Tensor
    kept: torch.Tensor
    budgets: torch.Tensor
    sel: torch.Tensor
    sel_off: torch.Tensor
    cu_seqlens: torch.Tensor
    positions: torch.Tensor
    hidden: torch.Tensor      # [T, d] bf16: packed input, then (after prefill) final hidden states


class ScenePipeline:
    """Buffers for scenes of N tiles x n_v tokens x d, and the run of one query."""

    def __init__(self, N, n_v, d, xdt, M, S, Q, knn_m, policy, model: DeviceModel | None = None,
                 max_T: int | None = None, device="cuda"):
        self.N, self.n_v, self.d, self.M, self.S, self.Q = N, n_v, d, M, S, Q
        self.xdt = abi.RIFT_BF16 if xdt in ("bf16", torch.bfloat16) else abi.RIFT_F32
        self.knn_m = knn_m
        self.m = min(knn_m, N - 1)
        self.policy = abi.make_policy(policy)
        # contextual tokens (the merge of Stage 2): at most floor(ctx_num c / ctx_den) per tile
        num, den = getattr(policy, "ctx_num", 0), getattr(policy, "ctx_den", 64)
        self.max_m = max([(num * c) // den for c in policy.C if c < n_v] + [0]) if num else 0
        self.model = model
        self.max_T = max_T if max_T is not None else N * (S + n_v + Q)
        self.max_len = S + n_v + Q
        dev = torch.device(device)
        f32, i32 = dict(dtype=torch.float32, device=dev), dict(dtype=torch.int32, device=dev)
        self.t = torch.empty(d, **f32)
        self.B = torch.empty(max(M, 1), d, **f32)
        self.token_scores = torch.empty(N, n_v, **f32)
        self.tile_s_raw = torch.empty(N, **f32)
        self.tile_s = torch.empty(N, **f32)
        self.nbr = torch.empty(max(N * self.m, 1), **i32)
        self.u = torch.empty(N, **f32)
        self.kept = torch.empty(N, **i32)
        self.n_kept = torch.zeros(1, **i32)
        self.budgets = torch.empty(N, **i32)
        self.sel = torch.empty(N * n_v, **i32)
        self.sel_off = torch.empty(N + 1, **i32)
        self.packed = torch.empty(self.max_T, d, dtype=torch.bfloat16, device=dev)
        self.cu = torch.empty(N + 1, **i32)
        self.positions = torch.empty(max(self.max_T, 1), **i32)
        self.T = torch.zeros(1, **i32)
        self.counts_host = torch.zeros(2, dtype=torch.int32, pin_memory=True)
        self.max_ctx = N * self.max_m
        self.ctx = torch.empty(max(self.max_ctx, 1), d, dtype=torch.bfloat16, device=dev) if self.max_m else None
        self.ctx_off = torch.zeros(N + 1, **i32) if self.max_m else None
        self.ctx_target = torch.empty(max(self.max_ctx, 1), **i32) if self.max_m else None
        self.ws_merge_bytes = abi.merge_workspace_bytes(N, n_v) if self.max_m else 0
        self.ws_merge = torch.empty(self.ws_merge_bytes, dtype=torch.uint8, device=dev) if self.max_m else None
        self.ws_score_bytes = abi.score_workspace_bytes(N, n_v, d, M)
        self.ws_score = torch.empty(self.ws_score_bytes, dtype=torch.uint8, device=dev)
        self.ws_prefill = None
        self.ws_prefill_bytes = 0
        self.device = dev

    def _prefill_ws(self, T, n_seq):
        """The prefill workspace for T rows and n_seq sequences of capacity (kept across queries)."""
        need = abi.prefill_workspace_bytes(self.model.struct, T, n_seq, self.max_len)
        if need > self.ws_prefill_bytes:
            self.ws_prefill = torch.empty(need, dtype=torch.uint8, device=self.device)
            self.ws_prefill_bytes = need
        return self.ws_prefill, need

    def select(self, X, embed, phrase_ids, bg_ids, p=None, n_templates=1, stream=None):
        """a1-a7: query prep, scoring, smoothing, pruning, budgets and token selection."""
        vocab = embed.shape[0]
        n_phrase = phrase_ids.numel() // n_templates
        abi.query_prep(embed, vocab, self.d, phrase_ids, n_templates, n_phrase, bg_ids if self.M else None,
                       self.M, self.t, self.B if self.M else None, stream)
        abi.score_tiles(X, self.xdt, self.N, self.n_v, self.d, self.t, self.B if self.M else None, self.M,
                        self.knn_m, self.token_scores, self.tile_s_raw, self.tile_s,
                        self.nbr if self.m > 0 else None, self.ws_score, self.ws_score_bytes, stream)
        abi.select_budgeted_tokens(self.token_scores, self.tile_s, self.N, self.n_v, p, self.policy, self.u,
                                   self.kept, self.n_kept, self.budgets, self.sel, self.sel_off, None, 0, stream)

    def features(self, X, kept_only=True, V=None, stream=None):
        """Predictor features (quadrant Eq. 1 scores, token-score max/mean/std) of the kept tiles
        (slot j = kept[j]) or of every tile; after select()."""
        out = torch.empty(self.N, abi.N_FEATURES, dtype=torch.float32, device=self.device)
        need = abi.features_workspace_bytes(self.N, self.d)
        ws = torch.empty(need, dtype=torch.uint8, device=self.device)
        abi.tile_features(X, self.xdt, self.N, self.n_v, self.d, self.t, self.B if self.M else None, self.M,
                          self.token_scores, self.kept if kept_only else None, self.n_kept if kept_only else None,
                          out, V, ws, need, stream)
        return out

    def merge(self, X, stream=None):
        """a7b (when the policy merges): the contextual tokens of every kept tile."""
        abi.merge_contextual(X, self.xdt, self.N, self.n_v, self.d, self.kept, self.n_kept, self.budgets, self.sel,
                             self.sel_off, self.ctx, self.max_ctx, self.ctx_off, self.ctx_target, self.ws_merge,
                             self.ws_merge_bytes, stream)

    def pack(self, X, embed, sys_ids, query_ids, stream=None, with_system=True):
        """a8: the packed batch, cu_seqlens and positions (without the system rows: the suffixes
        for a shared-prefix prefill)."""
        if self.max_m:
            self.merge(X, stream)
        S = self.S if with_system else 0
        abi.pack_ragged(X, self.xdt, self.N, self.n_v, self.d, self.kept, self.n_kept, self.sel, self.sel_off,
                        sys_ids if S else None, S, query_ids, self.Q, embed, embed.shape[0], self.packed, self.max_T,
                        self.cu, self.positions, self.T, stream, ctx=self.ctx, ctx_off=self.ctx_off)

    def run_shared_prefix(self, X, embed, phrase_ids, bg_ids, sys_ids, query_ids, p=None, stream=None):
        """The query with the system prompt prefilled once: packed suffixes (vision tokens + query)
        prefilled over its cache.  Returns (n_kept, suffix rows); self.packed holds the suffixes'
        final hidden states, self.prefix_hidden the prompt's."""
        self.select(X, embed, phrase_ids, bg_ids, p, stream=stream)
        self.pack(X, embed, sys_ids, query_ids, stream, with_system=False)
        m, S = self.model, self.S
        if not hasattr(self, "prefix_hidden"):
            self.prefix_hidden = torch.empty(S, self.d, dtype=torch.bfloat16, device=self.device)
            self.prefix_kv = torch.empty(m.dec.n_layers, 2, S, self.d, dtype=torch.float16, device=self.device)
        need = abi.prefill_shared_prefix_workspace_bytes(m.struct, self.max_T, self.N, self.max_len, S)
        if need > self.ws_prefill_bytes:
            self.ws_prefill = torch.empty(need, dtype=torch.uint8, device=self.device)
            self.ws_prefill_bytes = need
        abi.prefill_shared_prefix(m.struct, sys_ids, S, embed, embed.shape[0], self.prefix_hidden, self.prefix_kv,
                                  self.packed, self.T, self.cu, self.n_kept, self.max_len, self.positions, None,
                                  self.ws_prefill, self.ws_prefill_bytes, stream, max_T=self.max_T, max_seqs=self.N)
        return self.read_counts(stream)

    def _enqueue_counts(self, stream=None):
        """Copy (n_kept, T) into pinned host memory on `stream` once they are written, and record
        an event for counts() to wait on."""
        s = stream if stream is not None else torch.cuda.current_stream()
        with torch.cuda.stream(s):
            self.counts_host[0:1].copy_(self.n_kept, non_blocking=True)
            self.counts_host[1:2].copy_(self.T, non_blocking=True)
            self._counts_ev = torch.cuda.Event()
            self._counts_ev.record(s)

    def counts(self):
        """(n_kept, T) of the last query run with counts=False: waits only until its packing has
        finished (the prefill may still be running).  The next query of this pipeline overwrites
        them."""
        self._counts_ev.synchronize()
        return int(self.counts_host[0]), int(self.counts_host[1])

    def read_counts(self, stream=None):
        """Sync, check device error flags and read (n_kept, T) back to the host."""
        s = stream if stream is not None else torch.cuda.current_stream()
        self._enqueue_counts(s)
        abi.sync_status(s)
        return int(self.counts_host[0]), int(self.counts_host[1])

    def prefill(self, stream=None, kv_out=None, last_logits=None, counts=None):
        """a9: decoder prefill over the packed batch, in place, with the row and sequence counts
        the packing left on the device (capacities max_T and N), or with host counts
        counts = (n_seq, T) read back earlier, which are then also the capacities (so that the
        optional KV cache, fp16 [n_layers, 2, T, d], is sized for the rows it holds).  Optional
        last-token logits: fp32 [capacity, vocab]."""
        if counts is not None:
            n_seq, T = counts
            ws, need = self._prefill_ws(T, n_seq)
            abi.prefill_layers(self.model.struct, self.packed, T, self.cu, n_seq, self.max_len, self.positions, ws,
                               need, stream, kv_out=kv_out, last_logits=last_logits)
            return
        ws, need = self._prefill_ws(self.max_T, self.N)
        abi.prefill_layers(self.model.struct, self.packed, self.T, self.cu, self.n_kept, self.max_len,
                           self.positions, ws, need, stream, kv_out=kv_out, last_logits=last_logits,
                           max_T=self.max_T, max_seqs=self.N)

    def decode(self, kv_cache, T, n_seq, token_ids, embed, hidden_out=None, kv_new=None, logits=None,
               stream=None):
        """One decode step after the prefill: token_ids[i] appended to sequence i."""
        max_len = self.max_len + 1
        need = abi.decode_workspace_bytes(self.model.struct, n_seq, max_len)
        ws = torch.empty(max(need, 256), dtype=torch.uint8, device=self.device)
        abi.decode_step(self.model.struct, kv_cache, T, self.cu, n_seq, max_len, token_ids, embed, embed.shape[0],
                        hidden_out, kv_new, logits, ws, need, stream)

    def run_batch(self, queries, prefill=True, stream=None):
        """Several scene queries through one prefill: each query (a tuple X, embed, phrase_ids,
        bg_ids, sys_ids, query_ids) is scored, selected and packed after the rows of the ones
        before it (rift_pack_ragged_at), then the whole batch is prefilled at once.  Returns
        [(n_kept, T, first row, first sequence)] per query; self.batch_packed[:rows] holds the
        batch (final hidden states after the prefill), self.batch_cu and
        self.batch_positions its offsets and positions."""
        B = len(queries)
        cap_rows, cap_seq = B * self.max_T, B * self.N
        if getattr(self, "batch_cap", (0, 0)) < (cap_rows, cap_seq):
            dev, i32 = self.device, dict(dtype=torch.int32, device=self.device)
            self.batch_packed = torch.empty(cap_rows, self.d, dtype=torch.bfloat16, device=dev)
            self.batch_positions = torch.empty(cap_rows, **i32)
            self.batch_cu = torch.empty(cap_seq + 1, **i32)
            self.batch_cap = (cap_rows, cap_seq)
        out, row0, seq0 = [], 0, 0
        for (X, embed, phrase_ids, bg_ids, sys_ids, query_ids) in queries:
            self.select(X, embed, phrase_ids, bg_ids, stream=stream)
            if self.max_m:
                self.merge(X, stream)
            abi.pack_ragged(X, self.xdt, self.N, self.n_v, self.d, self.kept, self.n_kept, self.sel, self.sel_off,
                            sys_ids if self.S else None, self.S, query_ids, self.Q, embed, embed.shape[0],
                            self.batch_packed[row0:], cap_rows - row0, self.batch_cu[seq0:],
                            self.batch_positions[row0:], self.T, stream, ctx=self.ctx, ctx_off=self.ctx_off,
                            row_base=row0)
            n_kept, T = self.read_counts(stream)
            out.append((n_kept, T, row0, seq0))
            row0, seq0 = row0 + T, seq0 + n_kept
        if prefill and self.model is not None and row0 > 0:
            ws, need = self._prefill_ws(row0, seq0)
            abi.prefill_layers(self.model.struct, self.batch_packed, row0, self.batch_cu, seq0, self.max_len,
                               self.batch_positions, ws, need, stream)
        return out

    def run(self, X, embed, phrase_ids, bg_ids, sys_ids, query_ids, p=None, prefill=True, stream=None,
            counts=True):
        """One scene query, a1-a9, enqueued on `stream` with no host wait in between.  counts=True
        then waits for it, checks the device error flags and returns (n_kept, T); counts=False
        returns at once (None): counts() gives them once the packing has run."""
        self.select(X, embed, phrase_ids, bg_ids, p, stream=stream)
        self.pack(X, embed, sys_ids, query_ids, stream)
        self._enqueue_counts(stream)
        if prefill and self.model is not None:
            self.prefill(stream)
        if counts:
            abi.sync_status(stream)
            return self.counts()
        return None

    def result(self, n_kept, T) -> QueryResult:
        return QueryResult(n_kept, T, self.t, self.token_scores, self.tile_s_raw, self.tile_s,
                           self.nbr[:self.N * self.m].view(self.N, self.m), self.u, self.kept[:n_kept],
                           self.budgets[:n_kept], self.sel, self.sel_off[:n_kept + 1], self.cu[:n_kept + 1],
                           self.positions[:T], self.packed[:T])
