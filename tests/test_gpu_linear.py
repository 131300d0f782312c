"""The prefill's linear layer (rift_linear: tcgen05 GEMM with fused epilogues) against fp64
products of the same fp16 operands, on shapes with M, N and K tails and the 7B shapes."""
import pytest
import torch

from synth import rng

pytestmark = pytest.mark.gpu

# fp16 outputs carry one rounding (relative 2^-12); fp32 accumulation over K adds far less.
F16_TOL = 2e-3
F32_TOL = 1e-4


def _rand(shape, stream, scale=1.0):
    n = 1
    for s in shape:
        n *= s
    return (rng.normal_f32(5, rng.stream_id("linear", stream), n).view(*shape) * scale).to(torch.float16)


def _rel(g, o):
    return float((g.double() - o).abs().max() / o.abs().max())


# M >= 1024 runs on SM pairs (256 x 256 tiles): ragged last tiles whose second 128 rows or second
# 128 B rows lie wholly or partly outside the operands.
SHAPES = [(1, 256, 64), (128, 256, 64), (129, 264, 72), (200, 768, 256), (384, 256, 688), (333, 1024, 4096),
          (1000, 4096, 4096), (300, 12288, 4096), (1100, 264, 72), (2000, 640, 200), (4097, 768, 128),
          (1024, 4096, 4096)]


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_store_bf16(M, N, K, cuda, riftlib):
    A, W = _rand((M, K), 1), _rand((N, K), 2, 0.05)
    out = torch.empty(M, N, dtype=torch.float16, device=cuda)
    riftlib.linear(A.to(cuda), W.to(cuda), M, N, K, riftlib.RIFT_EPI_STORE_F16, out)
    riftlib.sync_status()
    ref = A.double() @ W.double().T
    assert _rel(out.cpu(), ref) < F16_TOL


@pytest.mark.parametrize("M,N,K", [(129, 264, 72), (384, 256, 688), (777, 4096, 4096), (257, 4096, 11008),
                                   (1500, 4096, 688), (1030, 264, 11008)])
def test_residual_f32(M, N, K, cuda, riftlib):
    A, W = _rand((M, K), 3), _rand((N, K), 4, 0.05)
    R0 = rng.normal_f32(5, 77, M * N).view(M, N)
    R = R0.to(cuda)
    riftlib.linear(A.to(cuda), W.to(cuda), M, N, K, riftlib.RIFT_EPI_RESID_F32, R)
    riftlib.sync_status()
    ref = R0.double() + A.double() @ W.double().T
    assert _rel(R.cpu(), ref) < F32_TOL


@pytest.mark.parametrize("M,F,K", [(96, 688, 256), (300, 1376, 688), (513, 11008, 4096), (1300, 1376, 688)])
def test_swiglu(M, F, K, cuda, riftlib):
    from paper_2609_29029_gb300 import interleave_gate_up
    A = _rand((M, K), 5)
    Wg, Wu = _rand((F, K), 6, 0.05), _rand((F, K), 7, 0.05)
    W = interleave_gate_up(Wg, Wu)
    out = torch.empty(M, F, dtype=torch.float16, device=cuda)
    riftlib.linear(A.to(cuda), W.to(cuda), M, 2 * F, K, riftlib.RIFT_EPI_SWIGLU, out)
    riftlib.sync_status()
    g = A.double() @ Wg.double().T
    u = A.double() @ Wu.double().T
    ref = g / (1 + torch.exp(-g)) * u
    assert _rel(out.cpu(), ref) < F16_TOL


def test_back_to_back_calls_reuse_nothing_stale(cuda, riftlib):
    # a big call followed by a small one: the persistent kernel's barriers start fresh each launch
    for M, N, K in [(2048, 4096, 4096), (3, 256, 64), (2048, 4096, 4096)]:
        A, W = _rand((M, K), 8), _rand((N, K), 9, 0.05)
        out = torch.empty(M, N, dtype=torch.float16, device=cuda)
        riftlib.linear(A.to(cuda), W.to(cuda), M, N, K, riftlib.RIFT_EPI_STORE_F16, out)
        riftlib.sync_status()
        assert _rel(out.cpu(), A.double() @ W.double().T) < F16_TOL
