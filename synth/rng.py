"""Counter-based random numbers that are bit-identical on CPU and GPU.

Every value is a pure function of (seed, stream, index), evaluated with torch
integer tensor ops whose intermediate values stay below 2**63, so the same bits
come out on any device.  Floating point enters only at the end, as one
correctly rounded fp32 multiply of an exactly representable integer, which
IEEE fixes on every device.

Hash: ``lowbias32`` (xorshift-multiply, constants 0x7feb352d / 0x846ca68b),
published by C. Wellons in the hash-prospector project.

This module holds no arithmetic of the method; it only makes inputs.
"""
from __future__ import annotations

import math

import torch

M32 = 0xFFFFFFFF
_C1 = 0x7FEB352D
_C2 = 0x846CA68B

# Irwin-Hall sum of four 16-bit uniforms: mean 4 * 65535/2, variance 4 * (2^32 - 1)/12.
_IH_MEAN = 131070
_IH_INV_STD = float(torch.tensor(1.0 / math.sqrt((2.0 ** 32 - 1.0) / 3.0), dtype=torch.float32))

CHUNK = 1 << 25


def lowbias32_int(x: int) -> int:
    """The hash on one Python int (reference form for tests)."""
    x &= M32
    x ^= x >> 16
    x = (x * _C1) & M32
    x ^= x >> 15
    x = (x * _C2) & M32
    x ^= x >> 16
    return x


def _mul32(x: torch.Tensor, m: int) -> torch.Tensor:
    # (x * m) mod 2^32 for 0 <= x < 2^32 without leaving int63: split x into 16-bit halves.
    lo = x & 0xFFFF
    hi = x >> 16
    return ((((hi * m) & 0xFFFF) << 16) + lo * m) & M32


def lowbias32(x: torch.Tensor) -> torch.Tensor:
    x = x ^ (x >> 16)
    x = _mul32(x, _C1)
    x = x ^ (x >> 15)
    x = _mul32(x, _C2)
    x = x ^ (x >> 16)
    return x


def stream_key(seed: int, stream: int) -> int:
    return lowbias32_int(lowbias32_int(seed * 0x9E3779B9 + 0x632BE5AB) ^ (stream & M32) ^ ((stream >> 32) * 0x85EBCA6B))


def stream_id(*parts) -> int:
    """Stable 64-bit stream id from a tuple of ints/strings (no Python hash())."""
    h = 0x12345678
    for p in parts:
        if isinstance(p, str):
            for ch in p.encode():
                h = lowbias32_int(h ^ ch)
        else:
            h = lowbias32_int(h ^ (int(p) & M32))
            h = lowbias32_int(h ^ ((int(p) >> 32) & M32))
    return h


def hash_u32(key: int, idx: torch.Tensor) -> torch.Tensor:
    """u32 hash of counters ``idx`` (int64, >= 0) under a stream key."""
    lo = idx & M32
    hi = idx >> 32
    return lowbias32(lo ^ lowbias32(hi ^ key))


def hash_u32_int(key: int, idx: int) -> int:
    return lowbias32_int((idx & M32) ^ lowbias32_int((idx >> 32) ^ key))


def normal_int(key: int, i: int) -> float:
    """Reference form of element ``i`` of ``normal_f32`` (pure Python, for tests)."""
    h0 = hash_u32_int(key, 2 * i)
    h1 = hash_u32_int(key, 2 * i + 1)
    s = (h0 & 0xFFFF) + (h0 >> 16) + (h1 & 0xFFFF) + (h1 >> 16)
    a = torch.tensor(float(s - _IH_MEAN), dtype=torch.float32)
    return float(a * torch.tensor(_IH_INV_STD, dtype=torch.float32))


def _normal_chunk(key: int, start: int, n: int, device) -> torch.Tensor:
    i = torch.arange(start, start + n, dtype=torch.int64, device=device)
    h0 = hash_u32(key, 2 * i)
    h1 = hash_u32(key, 2 * i + 1)
    s = (h0 & 0xFFFF) + (h0 >> 16) + (h1 & 0xFFFF) + (h1 >> 16)
    return (s - _IH_MEAN).to(torch.float32) * _IH_INV_STD


def normal_f32(seed: int, stream: int, n: int, device="cpu", offset: int = 0) -> torch.Tensor:
    """n approximately standard-normal fp32 values (Irwin-Hall-4, unit variance)."""
    key = stream_key(seed, stream)
    out = torch.empty(n, dtype=torch.float32, device=device)
    for s in range(0, n, CHUNK):
        m = min(CHUNK, n - s)
        out[s:s + m] = _normal_chunk(key, offset + s, m, device)
    return out


def uniform_f32(seed: int, stream: int, n: int, device="cpu") -> torch.Tensor:
    """n uniforms in [0, 1) with 24-bit resolution (exact in fp32)."""
    key = stream_key(seed, stream)
    i = torch.arange(n, dtype=torch.int64, device=device)
    return (hash_u32(key, i) >> 8).to(torch.float32) * (1.0 / (1 << 24))


def uniform_f64_host(seed: int, stream: int, n: int) -> list:
    """n uniforms in [0, 1) as Python floats (host-side parameters)."""
    key = stream_key(seed, stream)
    return [hash_u32_int(key, i) / 4294967296.0 for i in range(n)]


def sign_vector(seed: int, stream: int, d: int, device="cpu") -> torch.Tensor:
    """A vector of +-1/sqrt(d): exactly unit length in fp32 when d is a power of 4."""
    key = stream_key(seed, stream)
    i = torch.arange(d, dtype=torch.int64, device=device)
    bit = (hash_u32(key, i) >> 31).to(torch.float32)
    return (1.0 - 2.0 * bit) * (1.0 / math.sqrt(d))


def permutation_prefix(seed: int, stream: int, n: int, k: int) -> list:
    """The first k entries of a seeded permutation of range(n) (host ints)."""
    key = stream_key(seed, stream)
    keyed = sorted((hash_u32_int(key, i), i) for i in range(n))
    return [i for _, i in keyed[:k]]
