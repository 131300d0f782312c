"""The C-ABI library builds, loads and exports every entry point of include/rift.h; host-side
argument validation rejects bad calls before anything reaches a GPU.  No GPU needed."""
import ctypes as C
import re
from pathlib import Path

import pytest

HEADER = Path(__file__).resolve().parent.parent / "include" / "rift.h"


def declared_functions():
    text = re.sub(r"/\*.*?\*/", "", HEADER.read_text(), flags=re.S)
    names = re.findall(r"^[A-Za-z_][\w\s\*]*?\b(rift_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_hot_path_calls():
    names = declared_functions()
    for n in ("rift_query_prep", "rift_score_tiles", "rift_select_budgeted_tokens", "rift_pack_ragged",
              "rift_prefill_layers", "rift_sync_status"):
        assert n in names


def test_library_exports_every_declared_symbol(riftlib):
    lib = C.CDLL(str(riftlib.LIB_PATH))
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings(riftlib):
    assert riftlib.status_string(0) == "ok"
    assert riftlib.status_string(riftlib.RIFT_ERR_CAPACITY) == "output capacity exceeded"
    assert riftlib.abi_version() == 5


FAKE = 0x10000  # a 16-byte aligned non-null address; validation rejects before using it


def test_score_tiles_rejects_bad_shapes(riftlib):
    lib = riftlib.lib
    ws = riftlib.score_workspace_bytes(4, 576, 256, 8)
    assert ws > 0
    args = dict(X=FAKE, xdt=1, N=4, n_v=576, d=256, t=FAKE, B=FAKE, M=8, knn_m=6, r=FAKE, s0=FAKE, s1=FAKE,
                nbr=None, ws=FAKE, wsb=ws, st=0)

    def call(**kw):
        a = dict(args, **kw)
        return lib.rift_score_tiles(a["X"], a["xdt"], a["N"], a["n_v"], a["d"], a["t"], a["B"], a["M"], a["knn_m"],
                                    a["r"], a["s0"], a["s1"], a["nbr"], a["ws"], a["wsb"], a["st"])

    INV = riftlib.RIFT_ERR_INVALID
    assert call(N=0) == INV
    assert call(n_v=0) == INV and call(n_v=1025) == INV
    assert call(d=100) == INV and call(d=8256) == INV
    assert call(knn_m=-1) == INV and call(knn_m=17) == INV
    assert call(X=None) == INV and call(r=None) == INV
    assert call(X=FAKE + 4) == INV            # misaligned tokens
    assert call(wsb=ws - 1) == INV            # workspace too small
    assert call(ws=FAKE + 8) == INV           # workspace misaligned
    assert call(xdt=7) == INV
    assert call(M=1, B=None) == INV
    assert call(xdt=0, d=8192) == riftlib.RIFT_ERR_UNSUPPORTED


def _policy(riftlib, **kw):
    from synth import workloads as W
    p = riftlib.make_policy(W.RIFT_POLICY)
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def test_select_rejects_bad_policies(riftlib):
    lib = riftlib.lib

    def call(pol, N=4, n_v=576):
        return lib.rift_select_budgeted_tokens(FAKE, FAKE, N, n_v, None, C.byref(pol), FAKE, FAKE, FAKE, FAKE,
                                               FAKE, FAKE, None, 0, 0)

    INV = riftlib.RIFT_ERR_INVALID
    assert call(_policy(riftlib, tau=1.5)) == INV
    assert call(_policy(riftlib, tau=float("nan"))) == INV
    assert call(_policy(riftlib, n_c=0)) == INV and call(_policy(riftlib, n_c=9)) == INV
    p = _policy(riftlib)
    p.C[1], p.C[2] = p.C[2], p.C[1]          # not ascending
    assert call(p) == INV
    assert call(_policy(riftlib), n_v=288) == INV   # C holds 576 > n_v
    p = _policy(riftlib)
    p.alpha_pos[0] = float("inf")
    assert call(p) == INV
    assert call(_policy(riftlib), N=0) == INV


def test_pack_and_prefill_reject_bad_arguments(riftlib):
    lib = riftlib.lib
    INV = riftlib.RIFT_ERR_INVALID
    assert lib.rift_pack_ragged(FAKE, 1, 4, 576, 256, FAKE, FAKE, FAKE, FAKE, None, 8, FAKE, 16, FAKE, 1000, None,
                                None, FAKE, 100, FAKE, FAKE, FAKE, 0) == INV  # S > 0 without ids
    assert lib.rift_pack_ragged(FAKE, 1, 4, 576, 256, FAKE, FAKE, FAKE, FAKE, FAKE, 8, FAKE, 16, FAKE, 1000, None,
                                None, FAKE + 2, 100, FAKE, FAKE, FAKE, 0) == INV  # misaligned output
    assert lib.rift_pack_ragged(FAKE, 1, 4, 576, 256, FAKE, FAKE, FAKE, FAKE, FAKE, 8, FAKE, 16, FAKE, 1000, FAKE,
                                None, FAKE, 100, FAKE, FAKE, FAKE, 0) == INV  # contextual rows without offsets
    assert lib.rift_pack_ragged(FAKE, 1, 4, 576, 256, FAKE, FAKE, FAKE, FAKE, FAKE, 8, FAKE, 16, FAKE, 1000, FAKE + 8,
                                FAKE, FAKE, 100, FAKE, FAKE, FAKE, 0) == INV  # misaligned contextual rows
    assert lib.rift_pack_ragged_at(FAKE, 1, 4, 576, 256, FAKE, FAKE, FAKE, FAKE, FAKE, 8, FAKE, 16, FAKE, 1000, None,
                                   None, FAKE, 100, FAKE, FAKE, FAKE, -1, 0) == INV  # negative row base
    m = riftlib.Model()
    m.n_layers, m.d, m.n_heads, m.head_dim, m.ffn, m.eps, m.rope_theta = 2, 256, 4, 64, 688, 1e-6, 1e4
    assert lib.rift_prefill_workspace_bytes(C.byref(m), 100, 2, 64) == 0  # null weight arrays
    arr = (C.c_void_p * 2)(FAKE, FAKE)
    for f in ("w_qkv", "w_o", "w_gate_up", "w_down", "g_attn", "g_ffn"):
        setattr(m, f, arr)
    m.g_final = FAKE
    assert lib.rift_prefill_workspace_bytes(C.byref(m), 100, 2, 64) > 0
    m.head_dim = 96
    assert lib.rift_prefill_workspace_bytes(C.byref(m), 100, 2, 64) == 0
    m.head_dim, m.ffn = 64, 690
    assert lib.rift_prefill_layers(C.byref(m), FAKE, None, 10, FAKE, None, 1, 64, FAKE, None, None, FAKE, 1 << 30, 0) == INV
    m.ffn = 688
    # last-token logits need an output matrix; optional outputs must be 16-byte aligned
    assert lib.rift_prefill_layers(C.byref(m), FAKE, None, 10, FAKE, None, 1, 64, FAKE, None, FAKE, FAKE, 1 << 30, 0) == INV
    assert lib.rift_prefill_layers(C.byref(m), FAKE, None, 10, FAKE, None, 1, 64, FAKE, FAKE + 8, None, FAKE, 1 << 30, 0) == INV
    m.vocab, m.lm_head = 1000, FAKE
    assert lib.rift_prefill_layers(C.byref(m), FAKE, None, 10, FAKE, None, 1, 64, FAKE, None, FAKE + 4, FAKE, 1 << 30, 0) == INV
    m.vocab = 1001  # not a multiple of 8
    assert lib.rift_prefill_layers(C.byref(m), FAKE, None, 10, FAKE, None, 1, 64, FAKE, None, FAKE, FAKE, 1 << 30, 0) == INV
    m.vocab = 1000
    # rows without any sequence, negative capacities
    assert lib.rift_prefill_layers(C.byref(m), FAKE, FAKE, 10, FAKE, FAKE, 0, 64, FAKE, None, None, FAKE, 1 << 30, 0) == INV
    assert lib.rift_prefill_layers(C.byref(m), FAKE, FAKE, -1, FAKE, FAKE, 1, 64, FAKE, None, None, FAKE, 1 << 30, 0) == INV


def test_prefill_count_arguments(riftlib):
    """Host counts are their own capacities; a device count needs one (marshalling only)."""
    import torch
    assert riftlib._count(7, None, "T") == (None, 7)
    assert riftlib._count(7, 7, "T") == (None, 7)
    with pytest.raises(ValueError):
        riftlib._count(7, 9, "T")
    with pytest.raises(ValueError):
        riftlib._count(torch.zeros(1, dtype=torch.int32), None, "T")
    t = torch.zeros(1, dtype=torch.int32)
    assert riftlib._count(t, 9, "T") == (t.data_ptr(), 9)


def test_decode_rejects_bad_arguments(riftlib):
    lib = riftlib.lib
    INV = riftlib.RIFT_ERR_INVALID
    m = riftlib.Model()
    m.n_layers, m.d, m.n_heads, m.head_dim, m.ffn, m.eps, m.rope_theta = 2, 256, 4, 64, 688, 1e-6, 1e4
    arr = (C.c_void_p * 2)(FAKE, FAKE)
    for f in ("w_qkv", "w_o", "w_gate_up", "w_down", "g_attn", "g_ffn"):
        setattr(m, f, arr)
    m.g_final = FAKE
    ws = lib.rift_decode_workspace_bytes(C.byref(m), 3, 100)
    assert ws > 0
    assert lib.rift_decode_workspace_bytes(C.byref(m), 3, 40000) == 0     # max_len above 32768
    assert lib.rift_decode_workspace_bytes(C.byref(m), -1, 100) == 0

    def call(**kw):
        a = dict(kv=FAKE, T=10, cu=FAKE, n=3, max_len=100, ids=FAKE, embed=FAKE, ve=50, hid=FAKE, kvn=None,
                 lg=None, ws=FAKE, wsb=ws)
        a.update(kw)
        return lib.rift_decode_step(C.byref(m), a["kv"], a["T"], a["cu"], a["n"], a["max_len"], a["ids"], a["embed"],
                                    a["ve"], a["hid"], a["kvn"], a["lg"], a["ws"], a["wsb"], 0)

    assert call(kv=None) == INV and call(ids=None) == INV and call(embed=None) == INV
    assert call(max_len=0) == INV and call(max_len=40000) == INV and call(ve=0) == INV
    assert call(kv=FAKE + 2) == INV and call(hid=FAKE + 8) == INV
    assert call(lg=FAKE) == INV                   # logits without an output matrix
    assert call(wsb=ws - 1) == INV                # workspace too small


def test_query_prep_rejects_bad_arguments(riftlib):
    lib = riftlib.lib
    INV = riftlib.RIFT_ERR_INVALID
    assert lib.rift_query_prep(FAKE, 1000, 256, FAKE, 0, 16, FAKE, 8, FAKE, FAKE, 0) == INV
    assert lib.rift_query_prep(FAKE, 1000, 256, FAKE, 1, 16, None, 8, FAKE, FAKE, 0) == INV
    assert lib.rift_query_prep(FAKE, 1000, 200, FAKE, 1, 16, FAKE, 8, FAKE, FAKE, 0) == INV


def test_merge_and_policy_reject_bad_arguments(riftlib):
    lib = riftlib.lib
    INV = riftlib.RIFT_ERR_INVALID
    ws = lib.rift_merge_workspace_bytes(4, 576)
    assert ws > 0 and lib.rift_merge_workspace_bytes(0, 576) == 0 and lib.rift_merge_workspace_bytes(4, 2000) == 0

    def call(**kw):
        a = dict(X=FAKE, xdt=1, N=4, n_v=576, d=256, kept=FAKE, nk=FAKE, bud=FAKE, sel=FAKE, off=FAKE, ctx=FAKE,
                 max_ctx=100, coff=FAKE, tgt=FAKE, ws=FAKE, wsb=ws)
        a.update(kw)
        return lib.rift_merge_contextual(a["X"], a["xdt"], a["N"], a["n_v"], a["d"], a["kept"], a["nk"], a["bud"],
                                         a["sel"], a["off"], a["ctx"], a["max_ctx"], a["coff"], a["tgt"], a["ws"],
                                         a["wsb"], 0)

    assert call(X=None) == INV and call(coff=None) == INV and call(tgt=None) == INV
    assert call(ctx=None) == INV and call(max_ctx=-1) == INV and call(ctx=FAKE + 4) == INV
    assert call(wsb=ws - 1) == INV and call(xdt=5) == INV and call(d=100) == INV
    # policy: 0 <= ctx_num < ctx_den
    for num, den in ((-1, 64), (64, 64), (1, 0)):
        pol = _policy(riftlib, ctx_num=num, ctx_den=den)
        assert lib.rift_select_budgeted_tokens(FAKE, FAKE, 4, 576, None, C.byref(pol), FAKE, FAKE, FAKE, FAKE,
                                               FAKE, FAKE, None, 0, 0) == INV


def test_tile_features_reject_bad_arguments(riftlib):
    lib = riftlib.lib
    INV = riftlib.RIFT_ERR_INVALID
    ws = lib.rift_features_workspace_bytes(4, 256)
    assert ws > 0 and lib.rift_features_workspace_bytes(4, 100) == 0

    def call(**kw):
        a = dict(X=FAKE, xdt=1, N=4, n_v=576, d=256, t=FAKE, B=FAKE, M=8, r=FAKE, tiles=None, nt=None, f=FAKE,
                 V=None, ws=FAKE, wsb=ws)
        a.update(kw)
        return lib.rift_tile_features(a["X"], a["xdt"], a["N"], a["n_v"], a["d"], a["t"], a["B"], a["M"], a["r"],
                                      a["tiles"], a["nt"], a["f"], a["V"], a["ws"], a["wsb"], 0)

    assert call(X=None) == INV and call(r=None) == INV and call(f=None) == INV
    assert call(tiles=FAKE) == INV                       # a list without its count
    assert call(M=2, B=None) == INV and call(f=FAKE + 4) == INV and call(wsb=ws - 1) == INV
    assert call(n_v=200) == riftlib.RIFT_ERR_UNSUPPORTED  # not a square grid
    assert call(n_v=225) == riftlib.RIFT_ERR_UNSUPPORTED  # odd side: no quadrants


def test_noalloc_scoring_rejects_before_touching_the_gpu(riftlib):
    """The allocation-free scoring call checks its arguments, and that the scene's scratch fits the
    library's fixed array, before any CUDA call: these rejections need no GPU."""
    lib = riftlib.lib
    args = dict(X=FAKE, xdt=riftlib.RIFT_BF16, N=4, n_v=576, d=256, t=FAKE, B=FAKE, M=8, knn_m=6, r=FAKE, s0=FAKE,
                s1=FAKE, nbr=None, st=0)

    def call(**kw):
        a = dict(args, **kw)
        return lib.rift_score_tiles_noalloc(a["X"], a["xdt"], a["N"], a["n_v"], a["d"], a["t"], a["B"], a["M"],
                                            a["knn_m"], a["r"], a["s0"], a["s1"], a["nbr"], a["st"])

    INV = riftlib.RIFT_ERR_INVALID
    assert call(N=0) == INV and call(n_v=1025) == INV and call(d=100) == INV
    assert call(X=None) == INV and call(X=FAKE + 4) == INV and call(knn_m=17) == INV
    assert call(xdt=riftlib.RIFT_F32, d=8192) == riftlib.RIFT_ERR_UNSUPPORTED
    # 2000 tiles of 576 x 4096 need more scratch than the fixed array holds
    assert riftlib.score_workspace_bytes(2000, 576, 4096, 8) > riftlib.NOALLOC_SCORE_SCRATCH_BYTES
    assert call(N=2000, d=4096) == riftlib.RIFT_ERR_CAPACITY
