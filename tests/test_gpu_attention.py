"""rift_attention_varlen (tcgen05 varlen causal attention) against the oracle's fp64 attention
on the same fp16 q, k, v: lengths on both sides of every 128-row block boundary, both head
sizes, and logits large enough to force the rescaling of the running output."""
import numpy as np
import pytest
import torch

from oracle import rift_oracle as O
from synth import rng

pytestmark = pytest.mark.gpu

LENGTHS = [1, 2, 127, 128, 129, 255, 256, 257, 384, 385, 635]
# fp16 output (2^-11) and fp16 softmax weights; fp32 accumulation
TOL = 4e-3


def _run(riftlib, cuda, lengths, H, hd, q_scale):
    T = sum(lengths)
    d = H * hd
    x = rng.normal_f32(9, rng.stream_id("attn", H, hd, q_scale), T * 3 * d).view(T, 3, d)
    x[:, 0] *= q_scale
    qkv = x.reshape(T, 3 * d).to(torch.float16)
    cu = [0] + list(np.cumsum(lengths))
    cu_d = torch.tensor(cu, dtype=torch.int32, device=cuda)
    out = torch.full((T, d), float("nan"), dtype=torch.float16, device=cuda)
    need = riftlib.attention_workspace_bytes(T, len(lengths))
    ws = torch.empty(max(need, 256), dtype=torch.uint8, device=cuda)
    riftlib.attention_varlen(qkv.to(cuda), T, cu_d, len(lengths), H, hd, out, ws, need)
    riftlib.sync_status()
    return qkv, cu, out.cpu()


@pytest.mark.parametrize("H,hd,q_scale", [(4, 128, 1.0), (2, 64, 1.0), (4, 128, 6.0), (2, 64, 6.0)])
def test_attention_matches_fp64(H, hd, q_scale, cuda, riftlib):
    qkv, cu, out = _run(riftlib, cuda, LENGTHS, H, hd, q_scale)
    d = H * hd
    q3 = qkv.double().view(-1, 3, H, hd)
    worst = 0.0
    for j in range(len(cu) - 1):
        a, b = cu[j], cu[j + 1]
        ref = O.causal_attention(q3[a:b, 0], q3[a:b, 1], q3[a:b, 2]).reshape(b - a, d)
        got = out[a:b].double()
        assert torch.isfinite(got).all(), j
        err = float((got - ref).abs().max() / ref.abs().max())
        worst = max(worst, err)
        assert err < TOL, (j, b - a, err)
    print("worst", worst)


def test_attention_many_sequences_and_heads(cuda, riftlib):
    # more items than SMs: the persistent loop runs several items per CTA
    lengths = [131, 203, 347] * 30 + [635] * 4
    qkv, cu, out = _run(riftlib, cuda, lengths, 8, 128, 1.0)
    q3 = qkv.double().view(-1, 3, 8, 128)
    for j in (0, 1, 2, 45, 91, len(lengths) - 1):
        a, b = cu[j], cu[j + 1]
        ref = O.causal_attention(q3[a:b, 0], q3[a:b, 1], q3[a:b, 2]).reshape(b - a, 1024)
        assert float((out[a:b].double() - ref).abs().max() / ref.abs().max()) < TOL, j
