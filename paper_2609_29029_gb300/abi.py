"""ctypes binding of include/rift.h: the same call names, argument marshalling only.

Tensors are passed as raw device pointers (``tensor.data_ptr()``) and streams as raw
``cudaStream_t`` handles.  Every computation happens inside libriftgb.so; if the library is
missing this module raises at import time, there is no fallback.
"""
from __future__ import annotations

import ctypes as C
from pathlib import Path

import torch

LIB_PATH = Path(__file__).resolve().parent / "libriftgb.so"

RIFT_OK, RIFT_ERR_INVALID, RIFT_ERR_CAPACITY, RIFT_ERR_NONFINITE, RIFT_ERR_CUDA, RIFT_ERR_TIMEOUT, \
    RIFT_ERR_UNSUPPORTED, RIFT_ERR_BAD_ID = range(8)
RIFT_F32, RIFT_BF16 = 0, 1
RIFT_EPI_STORE_F16, RIFT_EPI_RESID_F32, RIFT_EPI_SWIGLU = 0, 1, 2
MAX_BUDGETS = 8


class RiftError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


class Policy(C.Structure):
    _fields_ = [("tau", C.c_float), ("n_c", C.c_int), ("C", C.c_int * MAX_BUDGETS),
                ("alpha_pos", C.c_float * MAX_BUDGETS), ("alpha_neg", C.c_float * MAX_BUDGETS),
                ("energy", C.c_float * MAX_BUDGETS), ("lam", C.c_float), ("ctx_num", C.c_int),
                ("ctx_den", C.c_int)]


class Model(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d", C.c_int), ("n_heads", C.c_int), ("head_dim", C.c_int),
                ("ffn", C.c_int), ("eps", C.c_float), ("rope_theta", C.c_float),
                ("w_qkv", C.POINTER(C.c_void_p)), ("w_o", C.POINTER(C.c_void_p)),
                ("w_gate_up", C.POINTER(C.c_void_p)), ("w_down", C.POINTER(C.c_void_p)),
                ("g_attn", C.POINTER(C.c_void_p)), ("g_ffn", C.POINTER(C.c_void_p)),
                ("g_final", C.c_void_p), ("vocab", C.c_int), ("lm_head", C.c_void_p)]


_vp, _i, _f, _sz = C.c_void_p, C.c_int, C.c_float, C.c_size_t

SIGNATURES = {
    "rift_abi_version": (_i, []),
    "rift_status_string": (C.c_char_p, [_i]),
    "rift_sync_status": (_i, [_vp]),
    "rift_query_prep": (_i, [_vp, _i, _i, _vp, _i, _i, _vp, _i, _vp, _vp, _vp]),
    "rift_score_workspace_bytes": (_sz, [_i, _i, _i, _i]),
    "rift_score_tiles": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _i, _i, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "rift_select_workspace_bytes": (_sz, [_i, _i]),
    "rift_select_budgeted_tokens": (_i, [_vp, _vp, _i, _i, _vp, C.POINTER(Policy), _vp, _vp, _vp, _vp, _vp,
                                         _vp, _vp, _sz, _vp]),
    "rift_pack_ragged": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _i, _vp, _i, _vp, _i, _vp, _vp,
                              _vp, _i, _vp, _vp, _vp, _vp]),
    "rift_pack_ragged_at": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _i, _vp, _i, _vp, _i, _vp, _vp,
                                 _vp, _i, _vp, _vp, _vp, _i, _vp]),
    "rift_features_workspace_bytes": (_sz, [_i, _i]),
    "rift_tile_features": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _i, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "rift_merge_workspace_bytes": (_sz, [_i, _i]),
    "rift_merge_contextual": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp, _i, _vp, _vp, _vp, _sz,
                                   _vp]),
    "rift_prefill_workspace_bytes": (_sz, [C.POINTER(Model), _i, _i, _i]),
    "rift_prefill_layers": (_i, [C.POINTER(Model), _vp, _vp, _i, _vp, _vp, _i, _i, _vp, _vp, _vp, _vp, _sz, _vp]),
    "rift_prefill_shared_prefix_workspace_bytes": (_sz, [C.POINTER(Model), _i, _i, _i, _i]),
    "rift_prefill_shared_prefix": (_i, [C.POINTER(Model), _vp, _i, _vp, _i, _vp, _vp, _vp, _vp, _i, _vp, _vp, _i, _i,
                                        _vp, _vp, _vp, _sz, _vp]),
    "rift_decode_workspace_bytes": (_sz, [C.POINTER(Model), _i, _i]),
    "rift_decode_step": (_i, [C.POINTER(Model), _vp, _i, _vp, _i, _i, _vp, _vp, _i, _vp, _vp, _vp, _vp, _sz,
                              _vp]),
    "rift_score_tiles_noalloc": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _i, _i, _vp, _vp, _vp, _vp, _vp]),
    "rift_score_shard_workspace_bytes": (_sz, [_i, _i, _i]),
    "rift_score_shard": (_i, [_vp, _i, _i, _i, _i, _vp, _vp, _i, _vp, _vp, _vp, _vp, _sz, _vp]),
    "rift_smooth_workspace_bytes": (_sz, [_i, _i, _i]),
    "rift_smooth_rows": (_i, [_vp, _vp, _i, _i, _i, _i, _i, _vp, _vp, _vp, _sz, _vp]),
    "rift_score_range": (_i, [_vp, _i, _vp, _vp]),
    "rift_select_budgeted_tokens_ranged": (_i, [_vp, _vp, _i, _i, _vp, _vp, C.POINTER(Policy), _vp, _vp, _vp, _vp,
                                                _vp, _vp, _vp]),
    "rift_linear": (_i, [_vp, _vp, _i, _i, _i, _i, _vp, _vp]),
    "rift_attention_workspace_bytes": (_sz, [_i, _i]),
    "rift_attention_varlen": (_i, [_vp, _i, _vp, _i, _i, _i, _vp, _vp, _sz, _vp]),
    "rift_check_wait_timeout": (_i, [_vp]),
    "rift_profile_enable": (None, [_i]),
    "rift_profile_read": (_i, [C.POINTER(C.c_double), C.POINTER(C.c_longlong), _i]),
    "rift_launch_count": (C.c_longlong, []),
}

PROF_CLASSES = ("gemm", "attention", "rmsnorm", "rope", "score", "select", "pack")


def _load():
    if not LIB_PATH.exists():
        raise ImportError(f"{LIB_PATH} is missing: build it first (python -m paper_2609_29029_gb300.build); "
                          "the Rift hot path has no CPU fallback")
    lib = C.CDLL(str(LIB_PATH))
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


lib = _load()


def status_string(s: int) -> str:
    return lib.rift_status_string(int(s)).decode()


def _check(status: int, where: str):
    if status != RIFT_OK:
        raise RiftError(status, where)


def ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def stream_handle(stream=None) -> int:
    if isinstance(stream, int):
        return stream
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def make_policy(policy) -> Policy:
    p = Policy()
    p.tau = policy.tau
    p.n_c = len(policy.C)
    for k, c in enumerate(policy.C):
        p.C[k] = c
        p.alpha_pos[k] = policy.alpha_pos[k]
        p.alpha_neg[k] = policy.alpha_neg[k]
        p.energy[k] = policy.energy[k]
    p.lam = policy.lam
    p.ctx_num = getattr(policy, "ctx_num", 0)
    p.ctx_den = getattr(policy, "ctx_den", 64)
    return p


def abi_version() -> int:
    return lib.rift_abi_version()


def sync_status(stream=None):
    _check(lib.rift_sync_status(stream_handle(stream)), "rift_sync_status")


def query_prep(embed, vocab, d, phrase_ids, n_templates, n_phrase, bg_ids, M, t, B, stream=None):
    _check(lib.rift_query_prep(ptr(embed), vocab, d, ptr(phrase_ids), n_templates, n_phrase, ptr(bg_ids), M,
                               ptr(t), ptr(B), stream_handle(stream)), "rift_query_prep")


def score_workspace_bytes(N, n_v, d, M) -> int:
    return lib.rift_score_workspace_bytes(N, n_v, d, M)


def score_tiles(X, xdt, N, n_v, d, t, B, M, knn_m, token_scores, tile_s_raw, tile_s, nbr, ws, ws_bytes,
                stream=None):
    _check(lib.rift_score_tiles(ptr(X), xdt, N, n_v, d, ptr(t), ptr(B), M, knn_m, ptr(token_scores),
                                ptr(tile_s_raw), ptr(tile_s), ptr(nbr), ptr(ws), ws_bytes, stream_handle(stream)),
           "rift_score_tiles")


def score_tiles_noalloc(X, xdt, N, n_v, d, t, B, M, knn_m, token_scores, tile_s_raw, tile_s, nbr, stream=None):
    """rift_score_tiles for callers without an allocator: scratch from the library's fixed array."""
    _check(lib.rift_score_tiles_noalloc(ptr(X), xdt, N, n_v, d, ptr(t), ptr(B), M, knn_m, ptr(token_scores),
                                        ptr(tile_s_raw), ptr(tile_s), ptr(nbr), stream_handle(stream)),
           "rift_score_tiles_noalloc")


NOALLOC_SCORE_SCRATCH_BYTES = 64 << 20


def score_shard_workspace_bytes(N_local, n_v, d) -> int:
    return lib.rift_score_shard_workspace_bytes(N_local, n_v, d)


def score_shard(X, xdt, N_local, n_v, d, t, B, M, token_scores, tile_s_raw, V, ws, ws_bytes, stream=None):
    _check(lib.rift_score_shard(ptr(X), xdt, N_local, n_v, d, ptr(t), ptr(B), M, ptr(token_scores), ptr(tile_s_raw),
                                ptr(V), ptr(ws), ws_bytes, stream_handle(stream)), "rift_score_shard")


def smooth_workspace_bytes(N, n_rows, d) -> int:
    return lib.rift_smooth_workspace_bytes(N, n_rows, d)


def smooth_rows(V, tile_s_raw, N, d, row0, n_rows, knn_m, tile_s, nbr, ws, ws_bytes, stream=None):
    _check(lib.rift_smooth_rows(ptr(V), ptr(tile_s_raw), N, d, row0, n_rows, knn_m, ptr(tile_s), ptr(nbr), ptr(ws),
                                ws_bytes, stream_handle(stream)), "rift_smooth_rows")


def score_range(tile_s, n, out, stream=None):
    _check(lib.rift_score_range(ptr(tile_s), n, ptr(out), stream_handle(stream)), "rift_score_range")


def select_budgeted_tokens_ranged(token_scores, tile_s, N, n_v, s_range, p, policy: Policy, u, kept, n_kept, budgets,
                                  sel, sel_off, stream=None):
    _check(lib.rift_select_budgeted_tokens_ranged(ptr(token_scores), ptr(tile_s), N, n_v, ptr(s_range), ptr(p),
                                                  C.byref(policy), ptr(u), ptr(kept), ptr(n_kept), ptr(budgets),
                                                  ptr(sel), ptr(sel_off), stream_handle(stream)),
           "rift_select_budgeted_tokens_ranged")


def select_workspace_bytes(N, n_v) -> int:
    return lib.rift_select_workspace_bytes(N, n_v)


def select_budgeted_tokens(token_scores, tile_s, N, n_v, p, policy: Policy, u, kept, n_kept, budgets, sel,
                           sel_off, ws, ws_bytes, stream=None):
    _check(lib.rift_select_budgeted_tokens(ptr(token_scores), ptr(tile_s), N, n_v, ptr(p), C.byref(policy),
                                           ptr(u), ptr(kept), ptr(n_kept), ptr(budgets), ptr(sel), ptr(sel_off),
                                           ptr(ws), ws_bytes, stream_handle(stream)),
           "rift_select_budgeted_tokens")


def pack_ragged(X, xdt, N, n_v, d, kept, n_kept, sel, sel_off, sys_ids, S, query_ids, Q, embed, vocab, packed,
                max_T, cu_seqlens, positions, T, stream=None, ctx=None, ctx_off=None, row_base=0):
    """rift_pack_ragged, or rift_pack_ragged_at with row_base > 0 (a later query of a batch:
    packed, cu_seqlens and positions are then that query's part of the batch buffers)."""
    if row_base:
        _check(lib.rift_pack_ragged_at(ptr(X), xdt, N, n_v, d, ptr(kept), ptr(n_kept), ptr(sel), ptr(sel_off),
                                       ptr(sys_ids), S, ptr(query_ids), Q, ptr(embed), vocab, ptr(ctx),
                                       ptr(ctx_off), ptr(packed), max_T, ptr(cu_seqlens), ptr(positions), ptr(T),
                                       row_base, stream_handle(stream)), "rift_pack_ragged_at")
        return
    _check(lib.rift_pack_ragged(ptr(X), xdt, N, n_v, d, ptr(kept), ptr(n_kept), ptr(sel), ptr(sel_off),
                                ptr(sys_ids), S, ptr(query_ids), Q, ptr(embed), vocab, ptr(ctx), ptr(ctx_off),
                                ptr(packed), max_T, ptr(cu_seqlens), ptr(positions), ptr(T), stream_handle(stream)),
           "rift_pack_ragged")


N_FEATURES = 7


def features_workspace_bytes(N, d) -> int:
    return lib.rift_features_workspace_bytes(N, d)


def tile_features(X, xdt, N, n_v, d, t, B, M, token_scores, tiles, n_tiles, features, V, ws, ws_bytes,
                  stream=None):
    _check(lib.rift_tile_features(ptr(X), xdt, N, n_v, d, ptr(t), ptr(B), M, ptr(token_scores), ptr(tiles),
                                  ptr(n_tiles), ptr(features), ptr(V), ptr(ws), ws_bytes, stream_handle(stream)),
           "rift_tile_features")


def merge_workspace_bytes(N, n_v) -> int:
    return lib.rift_merge_workspace_bytes(N, n_v)


def merge_contextual(X, xdt, N, n_v, d, kept, n_kept, budgets, sel, sel_off, ctx, max_ctx, ctx_off, ctx_target, ws,
                     ws_bytes, stream=None):
    _check(lib.rift_merge_contextual(ptr(X), xdt, N, n_v, d, ptr(kept), ptr(n_kept), ptr(budgets), ptr(sel),
                                     ptr(sel_off), ptr(ctx), max_ctx, ptr(ctx_off), ptr(ctx_target), ptr(ws),
                                     ws_bytes, stream_handle(stream)),
           "rift_merge_contextual")


def linear(A, W, M, N, K, epilogue, out, stream=None):
    _check(lib.rift_linear(ptr(A), ptr(W), M, N, K, epilogue, ptr(out), stream_handle(stream)), "rift_linear")


def attention_workspace_bytes(max_T, max_seqs) -> int:
    return lib.rift_attention_workspace_bytes(max_T, max_seqs)


def attention_varlen(qkv, T, cu_seqlens, n_seq, n_heads, head_dim, out, ws, ws_bytes, stream=None):
    _check(lib.rift_attention_varlen(ptr(qkv), T, ptr(cu_seqlens), n_seq, n_heads, head_dim, ptr(out), ptr(ws),
                                     ws_bytes, stream_handle(stream)), "rift_attention_varlen")


def prefill_workspace_bytes(model: Model, max_T, max_seqs, max_len) -> int:
    return lib.rift_prefill_workspace_bytes(C.byref(model), max_T, max_seqs, max_len)


def _count(c, cap, what):
    """A count argument of the prefill calls: a device int32 tensor (with its host capacity `cap`),
    or a host int, which is then both the count and the capacity (a NULL device pointer)."""
    if isinstance(c, int):
        if cap is not None and cap != c:
            raise ValueError(f"{what}: a host count is its own capacity; pass a device count to use {cap}")
        return None, c
    if cap is None:
        raise ValueError(f"{what}: a device count needs its host capacity")
    return ptr(c), cap


def prefill_layers(model: Model, hidden, T, cu_seqlens, n_seq, max_len, positions, ws, ws_bytes, stream=None,
                   kv_out=None, last_logits=None, max_T=None, max_seqs=None):
    """rift_prefill_layers.  T and n_seq: device int32 counts (with max_T and max_seqs, the host
    capacities), or host ints (then also the capacities)."""
    T_p, max_T = _count(T, max_T, "T")
    n_p, max_seqs = _count(n_seq, max_seqs, "n_seq")
    _check(lib.rift_prefill_layers(C.byref(model), ptr(hidden), T_p, max_T, ptr(cu_seqlens), n_p, max_seqs, max_len,
                                   ptr(positions), ptr(kv_out), ptr(last_logits), ptr(ws), ws_bytes,
                                   stream_handle(stream)),
           "rift_prefill_layers")


def prefill_shared_prefix_workspace_bytes(model: Model, max_T, max_seqs, max_len, S) -> int:
    return lib.rift_prefill_shared_prefix_workspace_bytes(C.byref(model), max_T, max_seqs, max_len, S)


def prefill_shared_prefix(model: Model, sys_ids, S, embed, vocab, prefix_hidden, prefix_kv, hidden, T, cu_seqlens,
                          n_seq, max_len, positions, last_logits, ws, ws_bytes, stream=None, max_T=None,
                          max_seqs=None):
    """rift_prefill_shared_prefix; T and n_seq as for prefill_layers."""
    T_p, max_T = _count(T, max_T, "T")
    n_p, max_seqs = _count(n_seq, max_seqs, "n_seq")
    _check(lib.rift_prefill_shared_prefix(C.byref(model), ptr(sys_ids), S, ptr(embed), vocab, ptr(prefix_hidden),
                                          ptr(prefix_kv), ptr(hidden), T_p, max_T, ptr(cu_seqlens), n_p, max_seqs,
                                          max_len, ptr(positions), ptr(last_logits), ptr(ws), ws_bytes,
                                          stream_handle(stream)),
           "rift_prefill_shared_prefix")


def decode_workspace_bytes(model: Model, n_seq, max_len) -> int:
    return lib.rift_decode_workspace_bytes(C.byref(model), n_seq, max_len)


def decode_step(model: Model, kv_cache, T, cu_seqlens, n_seq, max_len, token_ids, embed, vocab_embed,
                hidden_out, kv_new, logits, ws, ws_bytes, stream=None):
    _check(lib.rift_decode_step(C.byref(model), ptr(kv_cache), T, ptr(cu_seqlens), n_seq, max_len, ptr(token_ids),
                                ptr(embed), vocab_embed, ptr(hidden_out), ptr(kv_new), ptr(logits), ptr(ws), ws_bytes,
                                stream_handle(stream)),
           "rift_decode_step")


def check_wait_timeout(stream=None):
    _check(lib.rift_check_wait_timeout(stream_handle(stream)), "rift_check_wait_timeout")


def profile_enable(on: bool):
    lib.rift_profile_enable(1 if on else 0)


def profile_read() -> dict:
    """Per kernel class: (total ms, launches) recorded since profiling was enabled."""
    n = len(PROF_CLASSES)
    ms = (C.c_double * n)()
    cnt = (C.c_longlong * n)()
    _check(lib.rift_profile_read(ms, cnt, n), "rift_profile_read")
    return {k: (ms[i], cnt[i]) for i, k in enumerate(PROF_CLASSES)}


def launch_count() -> int:
    return lib.rift_launch_count()
