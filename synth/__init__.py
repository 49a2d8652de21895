"""Seeded synthetic inputs shared by the oracle tests, the GPU parity tests and bench.py.

This module holds no attention arithmetic.  It only draws numbers:

* ``bf16_normal`` -- i.i.d. N(0, 1) values rounded to bfloat16 (returned as the raw
  uint16 bit patterns), the input distribution of every workload.
* ``decode_lengths`` -- per-sequence KV lengths, uniform integers in a closed range.

The generator is counter based, so element ``i`` of a stream depends only on
``(seed, stream_id, i)`` and never on the platform, the thread count or the
torch/numpy version:

* SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014; constants as published by Vigna): the i-th output of a
  stream is ``mix(key + (i + 1) * GOLDEN)``.
* The stream key is ``mix(mix(seed) + stream_id)``.
* A uniform in the open interval (0, 1) is ``((x >> 11) + 0.5) * 2**-53``.
* Normals come from the Box-Muller transform: pair ``p`` uses uniforms ``2p`` and
  ``2p+1``; element ``2p`` takes the cosine branch, ``2p+1`` the sine branch.
* Rounding: float64 -> float32 (round to nearest even) -> bfloat16 (round to nearest
  even on the float32 bit pattern).

Stream ids used by the workloads: Q = 0, K = 1, V = 2, decode lengths = 3.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

__all__ = [
    "STREAM_Q", "STREAM_K", "STREAM_V", "STREAM_LENGTHS",
    "splitmix64_stream", "uniform01", "bf16_normal", "bf16_to_f32", "f32_to_bf16",
    "decode_lengths",
]

STREAM_Q, STREAM_K, STREAM_V, STREAM_LENGTHS = 0, 1, 2, 3

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22  # elements per worker task


def _mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser (in place on a uint64 array)."""
    z ^= z >> np.uint64(30)
    z *= _M1
    z ^= z >> np.uint64(27)
    z *= _M2
    z ^= z >> np.uint64(31)
    return z


def _mix_scalar(x: int) -> int:
    with np.errstate(over="ignore"):
        return int(_mix(np.array([x & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64))[0])


def _key(seed: int, stream_id: int) -> np.uint64:
    return np.uint64((_mix_scalar(seed) + stream_id) & 0xFFFFFFFFFFFFFFFF)


def splitmix64_stream(seed: int, stream_id: int, start: int, count: int) -> np.ndarray:
    """Outputs ``start .. start+count-1`` of stream ``(seed, stream_id)`` as uint64."""
    key = _key(seed, stream_id)
    with np.errstate(over="ignore"):
        ctr = np.arange(start + 1, start + count + 1, dtype=np.uint64)
        z = key + ctr * _GOLDEN
        return _mix(z)


def uniform01(bits: np.ndarray) -> np.ndarray:
    """Map uint64 words to float64 uniforms in the open interval (0, 1)."""
    return ((bits >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest even), returning the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bit patterns (uint16) to float32 exactly."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _normal_chunk(seed: int, stream_id: int, start: int, count: int) -> np.ndarray:
    """Elements ``start .. start+count-1`` (``start`` even) of the N(0,1) stream, as bf16 bits."""
    assert start % 2 == 0
    npairs = (count + 1) // 2
    bits = splitmix64_stream(seed, stream_id, start, 2 * npairs)
    u = uniform01(bits)
    u1, u2 = u[0::2], u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    t = (2.0 * math.pi) * u2
    z = np.empty(2 * npairs, dtype=np.float64)
    z[0::2] = r * np.cos(t)
    z[1::2] = r * np.sin(t)
    return f32_to_bf16(z[:count].astype(np.float32))


def bf16_normal(seed: int, stream_id: int, shape, *, start: int = 0, threads: int | None = None) -> np.ndarray:
    """N(0,1) values rounded to bf16, as a uint16 array of ``shape``.

    ``start`` selects a flat offset into the stream (even), so a slice of a large
    tensor can be regenerated without drawing the rest of it.
    """
    shape = (int(shape),) if np.isscalar(shape) else tuple(int(s) for s in shape)
    n = int(np.prod(shape)) if shape else 1
    if start % 2:
        raise ValueError("start must be even (normals are drawn in pairs)")
    out = np.empty(n, dtype=np.uint16)
    if n == 0:
        return out.reshape(shape)
    spans = [(s, min(_CHUNK, n - s)) for s in range(0, n, _CHUNK)]
    if len(spans) == 1:
        out[:] = _normal_chunk(seed, stream_id, start, n)
    else:
        nthreads = threads or min(len(spans), os.cpu_count() or 1)

        def work(span):
            s, c = span
            out[s:s + c] = _normal_chunk(seed, stream_id, start + s, c)

        with ThreadPoolExecutor(max_workers=nthreads) as ex:
            list(ex.map(work, spans))
    return out.reshape(shape)


def decode_lengths(seed: int, batch: int, lo: int, hi: int) -> np.ndarray:
    """``batch`` KV lengths, uniform integers in the closed range [lo, hi] (stream 3)."""
    if hi < lo:
        raise ValueError("hi < lo")
    u = uniform01(splitmix64_stream(seed, STREAM_LENGTHS, 0, batch))
    span = hi - lo + 1
    return (lo + np.minimum(np.floor(u * span), span - 1)).astype(np.int32)
