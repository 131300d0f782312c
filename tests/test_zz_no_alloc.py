"""rift_score_tiles_noalloc, the scoring entry point for callers that cannot allocate device
memory (programs whose device memory is fixed before they start, plug-ins without an allocator).
It takes its scratch from an array compiled into the library; its results must match
rift_score_tiles, which uses a caller-provided workspace, call after call.

This file is collected last on purpose: it runs after every other test, and alone.
"""
import pytest
import torch

from synth import workloads as W

import parity as P

pytestmark = pytest.mark.gpu


def _scene(wl, device):
    sc = W.make_scene(wl.scene, wl.decoder.vocab, device)
    return sc


def _outputs(wl, device):
    s = wl.scene
    f32 = dict(dtype=torch.float32, device=device)
    m = min(wl.knn_m, s.N - 1)
    return dict(r=torch.full((s.N, s.n_v), float("nan"), **f32), s0=torch.full((s.N,), float("nan"), **f32),
                s1=torch.full((s.N,), float("nan"), **f32),
                nbr=torch.full((max(s.N * m, 1),), -7, dtype=torch.int32, device=device))


def _query(abi, sc, wl, device):
    s = wl.scene
    i32 = dict(dtype=torch.int32, device=device)
    t = torch.empty(s.d, dtype=torch.float32, device=device)
    B = torch.empty(s.M, s.d, dtype=torch.float32, device=device)
    abi.query_prep(sc.embed, wl.decoder.vocab, s.d, torch.tensor(sc.query_ids, **i32), 1, s.Q,
                   torch.tensor(sc.bg_ids, **i32), s.M, t, B)
    return t, B


def _score_both(abi, wl, sc, device):
    s = wl.scene
    xdt = abi.RIFT_BF16 if s.x_dtype == "bf16" else abi.RIFT_F32
    t, B = _query(abi, sc, wl, device)
    ref, got = _outputs(wl, device), _outputs(wl, device)
    need = abi.score_workspace_bytes(s.N, s.n_v, s.d, s.M)
    ws = torch.empty(need, dtype=torch.uint8, device=device)
    abi.score_tiles(sc.X, xdt, s.N, s.n_v, s.d, t, B, s.M, wl.knn_m, ref["r"], ref["s0"], ref["s1"], ref["nbr"],
                    ws, need)
    abi.score_tiles_noalloc(sc.X, xdt, s.N, s.n_v, s.d, t, B, s.M, wl.knn_m, got["r"], got["s0"], got["s1"],
                            got["nbr"])
    abi.sync_status()
    return ref, got


def _check(ref, got):
    assert P.rel_err_rows(got["r"].cpu().numpy(), ref["r"].cpu().numpy()) < P.SCORE_RTOL
    assert P.max_abs_rel(got["s0"].cpu(), ref["s0"].cpu()) < P.SCORE_RTOL
    assert P.max_abs_rel(got["s1"].cpu(), ref["s1"].cpu()) < P.SCORE_RTOL
    assert torch.equal(got["nbr"].cpu(), ref["nbr"].cpu())


def test_noalloc_scoring_matches_workspace_scoring_twice_in_a_row(cuda, riftlib):
    # Two different scenes back to back: the second call must not see the first call's scratch.
    wl_a = W.Workload("noalloc_a", W.SceneSpec(N=64, d=4096, x_dtype="bf16"), W.LLAVA7B, W.RIFT_POLICY)
    wl_b = P.SMALL24
    for wl in (wl_a, wl_b):
        sc = _scene(wl, cuda)
        ref, got = _score_both(riftlib, wl, sc, cuda)
        _check(ref, got)


def test_noalloc_tensor_core_gram_branch_twice_in_a_row(cuda, riftlib):
    # 1100 tiles: the kNN's Gram product over its largest scene that fits the array (at d = 256),
    # with its split operands, tensor maps, split-K partials and the Gram matrix itself all inside
    # the fixed array.
    wl = W.Workload("noalloc_gram", W.SceneSpec(N=1100, d=256, x_dtype="bf16"), W.LLAVA7B, W.RIFT_POLICY)
    s = wl.scene
    assert riftlib.score_workspace_bytes(s.N, s.n_v, s.d, s.M) <= riftlib.NOALLOC_SCORE_SCRATCH_BYTES
    sc = _scene(wl, cuda)
    for _ in range(2):
        ref, got = _score_both(riftlib, wl, sc, cuda)
        _check(ref, got)


class _Driver:
    """The few CUDA driver calls the second-context test needs, through ctypes."""

    def __init__(self):
        import ctypes
        self.C = ctypes
        self.lib = ctypes.CDLL("libcuda.so.1")

    def __call__(self, name, *args):
        rc = getattr(self.lib, name)(*args)
        assert rc == 0, f"{name} returned {rc}"

    def alloc_copy(self, host_bytes):
        C = self.C
        p = C.c_uint64(0)
        self("cuMemAlloc_v2", C.byref(p), C.c_size_t(max(len(host_bytes), 16)))
        if host_bytes:
            buf = C.create_string_buffer(host_bytes, len(host_bytes))
            self("cuMemcpyHtoD_v2", p, buf, C.c_size_t(len(host_bytes)))
        return p.value

    def read(self, dptr, nbytes):
        C = self.C
        buf = C.create_string_buffer(nbytes)
        self("cuMemcpyDtoH_v2", buf, C.c_uint64(dptr), C.c_size_t(nbytes))
        return buf.raw


def test_noalloc_in_a_second_context_of_the_device(cuda, riftlib):
    # A host that drives the GPU through its own driver-API context (not the runtime's primary
    # context) gets its own copy of the fixed array at another address: the call must look the
    # address up in the context that is current, and the primary context must keep working after.
    import numpy as np
    wl = P.SMALL24
    s = wl.scene
    sc = _scene(wl, cuda)
    xdt = riftlib.RIFT_BF16 if s.x_dtype == "bf16" else riftlib.RIFT_F32
    ref, _ = _score_both(riftlib, wl, sc, cuda)
    t, B = _query(riftlib, sc, wl, cuda)
    host = {k: v.cpu().numpy() for k, v in dict(X=sc.X, t=t, B=B).items()}
    want = {k: v.cpu().numpy() for k, v in ref.items()}
    torch.cuda.synchronize()
    drv = _Driver()
    C = drv.C
    drv("cuInit", 0)
    dev, ctx = C.c_int(0), C.c_void_p(0)
    drv("cuDeviceGet", C.byref(dev), 0)
    drv("cuCtxCreate_v2", C.byref(ctx), 0, dev)  # created and made current on this thread
    try:
        d_in = {k: drv.alloc_copy(np.ascontiguousarray(v).tobytes()) for k, v in host.items()}
        d_out = {k: drv.alloc_copy(bytes(v.nbytes)) for k, v in want.items()}
        status = riftlib.lib.rift_score_tiles_noalloc(d_in["X"], xdt, s.N, s.n_v, s.d, d_in["t"], d_in["B"], s.M,
                                                      wl.knn_m, d_out["r"], d_out["s0"], d_out["s1"], d_out["nbr"],
                                                      None)
        assert status == riftlib.RIFT_OK
        drv("cuCtxSynchronize")
        assert riftlib.lib.rift_sync_status(None) == riftlib.RIFT_OK
        got = {k: np.frombuffer(drv.read(d_out[k], v.nbytes), dtype=v.dtype).reshape(v.shape) for k, v in want.items()}
        for p in list(d_in.values()) + list(d_out.values()):
            drv("cuMemFree_v2", C.c_uint64(p))
    finally:
        popped = C.c_void_p(0)
        drv("cuCtxPopCurrent_v2", C.byref(popped))
        drv("cuCtxDestroy_v2", ctx)
    assert P.rel_err_rows(got["r"], want["r"]) < P.SCORE_RTOL
    assert P.max_abs_rel(torch.from_numpy(got["s0"].copy()), torch.from_numpy(want["s0"])) < P.SCORE_RTOL
    assert P.max_abs_rel(torch.from_numpy(got["s1"].copy()), torch.from_numpy(want["s1"])) < P.SCORE_RTOL
    assert np.array_equal(got["nbr"], want["nbr"])
    # back in the primary context: its own array, its own address
    ref2, got2 = _score_both(riftlib, wl, sc, cuda)
    _check(ref2, got2)


def test_noalloc_rejects_scenes_larger_than_its_array(cuda, riftlib):
    N, n_v, d, M = 2000, 576, 4096, 8
    assert riftlib.score_workspace_bytes(N, n_v, d, M) > riftlib.NOALLOC_SCORE_SCRATCH_BYTES
    x = torch.empty(16, dtype=torch.bfloat16, device=cuda)
    f = torch.empty(16, dtype=torch.float32, device=cuda)
    status = riftlib.lib.rift_score_tiles_noalloc(x.data_ptr(), riftlib.RIFT_BF16, N, n_v, d, f.data_ptr(),
                                                  f.data_ptr(), M, 6, f.data_ptr(), f.data_ptr(), f.data_ptr(),
                                                  None, 0)
    assert status == riftlib.RIFT_ERR_CAPACITY
