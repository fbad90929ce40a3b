"""Counter-based seeded random numbers shared by the oracle side and the CUDA side.

This module draws numbers only; it contains none of the verification step's
arithmetic.  Everything is built on SplitMix64 (Steele, Lea and Flood,
"Fast splittable pseudorandom number generators", OOPSLA 2014; the mixing
constants are those of Vigna's public-domain splitmix64.c).  Output n of the
stream with key ``k`` is ``mix(k + (n + 1) * 0x9E3779B97F4A7C15)``, so any
element can be computed on its own and the same code runs on CPU and CUDA
tensors (torch int64 arithmetic wraps modulo 2**64).

Normal variates use the Box-Muller transform (Box and Muller, 1958): element n
takes the uniforms of counters 2n and 2n+1 and keeps the cosine branch.
"""

from __future__ import annotations

import math

import torch

GOLDEN = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

# Elements generated per chunk, to bound temporaries on large tensors.
CHUNK = 1 << 24


def _s64(x: int) -> int:
    """Python int (mod 2**64) -> the signed int64 with the same bits."""
    x &= MASK64
    return x - (1 << 64) if x >= (1 << 63) else x


def _srl(z: torch.Tensor, k: int) -> torch.Tensor:
    """Logical right shift of int64 bits."""
    return (z >> k) & ((1 << (64 - k)) - 1)


def splitmix64_scalar(key: int, n: int) -> int:
    """Output n of the SplitMix64 stream with state ``key`` (pure Python)."""
    z = (key + (n + 1) * GOLDEN) & MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def splitmix64(key: int, counters: torch.Tensor) -> torch.Tensor:
    """Outputs ``counters`` of the stream with state ``key``, as int64 bits."""
    z = counters.to(torch.int64) * _s64(GOLDEN) + _s64(key + GOLDEN)
    z = (z ^ _srl(z, 30)) * _s64(MIX1)
    z = (z ^ _srl(z, 27)) * _s64(MIX2)
    return z ^ _srl(z, 31)


def derive_key(seed: int, tag: int) -> int:
    """Independent stream key for (seed, tag): two SplitMix64 steps."""
    return splitmix64_scalar(splitmix64_scalar(seed & MASK64, tag & MASK64), 0)


def uniform(key: int, n: int, device="cpu", offset: int = 0) -> torch.Tensor:
    """n float64 uniforms in (0, 1): ((z >> 11) + 0.5) * 2**-53."""
    out = torch.empty(n, dtype=torch.float64, device=device)
    for s in range(0, n, CHUNK):
        e = min(n, s + CHUNK)
        c = torch.arange(offset + s, offset + e, dtype=torch.int64, device=device)
        out[s:e] = (_srl(splitmix64(key, c), 11).to(torch.float64) + 0.5) * (2.0 ** -53)
    return out


def uint64(key: int, n: int, device="cpu", offset: int = 0) -> torch.Tensor:
    """n raw outputs (int64 bits)."""
    c = torch.arange(offset, offset + n, dtype=torch.int64, device=device)
    return splitmix64(key, c)


def below(key: int, n: int, bound: int, device="cpu", offset: int = 0) -> torch.Tensor:
    """n integers in [0, bound): floor(u * bound) with u from ``uniform``."""
    u = uniform(key, n, device=device, offset=offset)
    return torch.clamp((u * bound).floor().to(torch.int64), max=bound - 1)


def normal(key: int, n: int, device="cpu") -> torch.Tensor:
    """n float64 N(0,1) variates (Box-Muller, cosine branch)."""
    out = torch.empty(n, dtype=torch.float64, device=device)
    half = CHUNK // 2
    for s in range(0, n, half):
        e = min(n, s + half)
        c = torch.arange(2 * s, 2 * e, dtype=torch.int64, device=device)
        u = (_srl(splitmix64(key, c), 11).to(torch.float64) + 0.5) * (2.0 ** -53)
        u1, u2 = u[0::2], u[1::2]
        out[s:e] = torch.sqrt(-2.0 * torch.log(u1)) * torch.cos((2.0 * math.pi) * u2)
    return out


def round_to(x: torch.Tensor, dtype: torch.dtype) -> torch.Tensor:
    """float64 -> float32 (round to nearest even) -> ``dtype`` (round to nearest even)."""
    x32 = x.to(torch.float32)
    return x32 if dtype == torch.float32 else x32.to(dtype)
