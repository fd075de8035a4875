"""Seeded synthetic inputs shared by the CUDA path's tests/bench and by the oracle's tests.

This module only draws numbers. It holds none of the scoring arithmetic (no linear
algebra, no softmax, no advantage estimation), so both sides of a parity test can take
their inputs from it without sharing any of the computation under test.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
generators", OOPSLA 2014) in counter form, i.e. draw i of stream `seed` is
mix(seed_state + (i + 1) * 0x9E3779B97F4A7C15). Uniforms take the top 53 bits.
Normals use the Box-Muller transform in float32: each 64-bit draw gives two 32-bit
uniforms (u1, u2) and two normals, r cos(2 pi u2) and r sin(2 pi u2), r = sqrt(-2 ln u1).
bf16 values are produced by rounding the fp32 value to nearest-even on the upper 16 bits.

Everything returned is numpy: bf16 tensors as uint16 bit patterns, fp32 as float32,
integer ids/lengths as int32.
"""
from __future__ import annotations

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22


def _splitmix64(seed: int, start: int, n: int) -> np.ndarray:
    """Counter-based SplitMix64 outputs for indices start .. start+n-1 of stream `seed`."""
    with np.errstate(over="ignore"):
        base = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) * _GOLDEN
        z = np.arange(start + 1, start + n + 1, dtype=np.uint64)
        z *= _GOLDEN
        z += base
        z ^= z >> np.uint64(30)
        z *= _M1
        z ^= z >> np.uint64(27)
        z *= _M2
        z ^= z >> np.uint64(31)
    return z


def uniform(seed: int, n: int) -> np.ndarray:
    """n doubles uniform in (0, 1), never exactly 0 (safe for log)."""
    out = np.empty(n, dtype=np.float64)
    for s in range(0, n, _CHUNK):
        m = min(_CHUNK, n - s)
        z = _splitmix64(seed, s, m)
        out[s:s + m] = ((z >> np.uint64(11)).astype(np.float64) + 0.5) * (1.0 / 9007199254740992.0)
    return out


def normal(seed: int, n: int, std: float = 1.0) -> np.ndarray:
    """n float32 draws from N(0, std^2) (Box-Muller, two normals per 64-bit draw)."""
    out = np.empty(2 * ((n + 1) // 2), dtype=np.float32)
    half = out.size // 2
    scale = np.float32(1.0 / 4294967296.0)
    for s in range(0, half, _CHUNK):
        m = min(_CHUNK, half - s)
        z = _splitmix64(seed, s, m)
        u1 = ((z >> np.uint64(32)).astype(np.float32) + np.float32(0.5)) * scale
        u2 = ((z & np.uint64(0xFFFFFFFF)).astype(np.float32) + np.float32(0.5)) * scale
        np.log(u1, out=u1)
        u1 *= np.float32(-2.0)
        np.sqrt(u1, out=u1)
        u1 *= np.float32(std)
        u2 *= np.float32(2.0 * np.pi)
        out[2 * s:2 * (s + m):2] = u1 * np.cos(u2)
        out[2 * s + 1:2 * (s + m):2] = u1 * np.sin(u2)
    return out[:n]


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest, ties to even); returns uint16 bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16(seed: int, shape, std: float = 1.0) -> np.ndarray:
    """bf16 bit patterns (uint16) of N(0, std^2) draws, in C order of `shape`."""
    n = int(np.prod(shape))
    return f32_to_bf16_bits(normal(seed, n, std).astype(np.float32)).reshape(shape)


def normal_f32(seed: int, shape, std: float = 1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return normal(seed, n, std).astype(np.float32).reshape(shape)


def randint(seed: int, shape, low: int, high: int) -> np.ndarray:
    """int32 uniform in [low, high) by 64-bit multiply-shift (Lemire) on SplitMix64 output."""
    n = int(np.prod(shape))
    span = high - low
    assert 0 < span < (1 << 31)
    out = np.empty(n, dtype=np.int64)
    for s in range(0, n, _CHUNK):
        m = min(_CHUNK, n - s)
        hi32 = (_splitmix64(seed, s, m) >> np.uint64(32)).astype(np.uint64)
        with np.errstate(over="ignore"):
            out[s:s + m] = ((hi32 * np.uint64(span)) >> np.uint64(32)).astype(np.int64)
    return (out + low).astype(np.int32).reshape(shape)


def tensor_seed(config: int, index: int) -> int:
    """Stream id of input tensor `index` of workload number `config`."""
    return 1000 * config + index
