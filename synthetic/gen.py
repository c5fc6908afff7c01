"""Seeded synthetic inputs shared by the oracle tests, the GPU parity tests and the bench.

This module holds none of the attention method's arithmetic: it only draws
reproducible random numbers and stores them as bf16 bit patterns.  Both the CPU
oracle and the CUDA path receive the same arrays from here, so neither side ever
generates its own inputs.

Generator (published definitions, written out here):
  * splitmix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
    generators", OOPSLA 2014; the 64-bit finaliser constants of Vigna's
    splitmix64.c).  Used counter-style: output i of the stream with key ``k`` is
    ``mix(k + (i + 1) * 0x9E3779B97F4A7C15)``.
  * Box-Muller transform (Box & Muller 1958) in float64: a pair of uniforms
    u1 in (0, 1], u2 in [0, 1) gives r*cos(2*pi*u2), r*sin(2*pi*u2) with
    r = sqrt(-2 ln u1).
  * Storage: float64 -> float32 (numpy, round to nearest even) -> bf16 by round
    to nearest even on the float32 bit pattern.  The bf16 bit patterns are the
    inputs; both implementations decode them exactly.

The per-tensor key is FNV-1a-64 of ``"<workload>/<tensor>"`` mixed with the seed,
so every tensor of every workload has its own independent stream.
"""
from __future__ import annotations

import concurrent.futures as cf
import os

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 20


def _mix(z: np.ndarray) -> np.ndarray:
    """splitmix64 output finaliser on a uint64 array (wrapping arithmetic)."""
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def fnv1a64(text: str) -> int:
    h = 0xCBF29CE484222325
    for b in text.encode("utf-8"):
        h ^= b
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def tensor_key(workload: str, tensor: str, seed: int = 0) -> int:
    """64-bit stream key for one named tensor of one workload."""
    base = np.array([fnv1a64(f"{workload}/{tensor}") ^ (seed & 0xFFFFFFFFFFFFFFFF)],
                    dtype=np.uint64)
    return int(_mix(base)[0])


def splitmix64_stream(key: int, start: int, count: int) -> np.ndarray:
    """Outputs ``start .. start+count-1`` of the splitmix64 stream with state ``key``."""
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(np.uint64(key) + idx * _GOLDEN)


def _mix_inplace(z: np.ndarray) -> None:
    z ^= z >> np.uint64(30)
    z *= _M1
    z ^= z >> np.uint64(27)
    z *= _M2
    z ^= z >> np.uint64(31)


def _normal_pairs(key: int, p0: int, p1: int, out: np.ndarray, n: int) -> None:
    """Box-Muller pairs p0..p1-1 (stream outputs 2p and 2p+1) into out[2*p0 : min(n, 2*p1)]."""
    two53 = float(2 ** 53)
    with np.errstate(over="ignore"):
        c = np.arange(2 * p0 + 1, 2 * p1 + 1, 2, dtype=np.uint64)  # counter of output 2p
        z1 = c * _GOLDEN
        z1 += np.uint64(key)
        _mix_inplace(z1)
        c += np.uint64(1)
        c *= _GOLDEN
        c += np.uint64(key)
        _mix_inplace(c)
    z1 >>= np.uint64(11)
    c >>= np.uint64(11)
    r = z1.astype(np.float64)
    r += 1.0
    r /= two53                      # u1 in (0, 1]
    t = c.astype(np.float64)
    t *= 2.0 * np.pi / two53        # 2*pi*u2 (scaling by 2^-53 is exact)
    np.log(r, out=r)
    r *= -2.0
    np.sqrt(r, out=r)
    lo, hi = 2 * p0, min(n, 2 * p1)
    m = p1 - p0
    if hi - lo == 2 * m:
        out[lo:hi:2] = r * np.cos(t)
        out[lo + 1:hi:2] = r * np.sin(t)
    else:
        pair = np.empty(2 * m)
        pair[0::2] = r * np.cos(t)
        pair[1::2] = r * np.sin(t)
        out[lo:hi] = pair[: hi - lo]


def normal_f64(key: int, n: int) -> np.ndarray:
    """``n`` standard normal float64 values (Box-Muller on counter-based splitmix64).

    Value 2p is r*cos(2*pi*u2) and value 2p+1 is r*sin(2*pi*u2), where u1 and u2
    come from stream outputs 2p and 2p+1.  Chunks are independent, so they are
    evaluated on a few threads (numpy releases the GIL); the result does not
    depend on the chunking.
    """
    out = np.empty(n, dtype=np.float64)
    npairs = (n + 1) // 2
    bounds = [(p0, min(npairs, p0 + _CHUNK)) for p0 in range(0, npairs, _CHUNK)]
    if len(bounds) <= 1:
        for p0, p1 in bounds:
            _normal_pairs(key, p0, p1, out, n)
        return out
    workers = max(1, min(8, (os.cpu_count() or 1), len(bounds)))
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(lambda b: _normal_pairs(key, b[0], b[1], out, n), bounds))
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit pattern (uint16), round to nearest even.  Finite inputs only."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    # no uint32 overflow for finite inputs: the largest pattern 0xFF7FFFFF + 0x8000 fits
    u = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (u >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit pattern (uint16) -> float32, exact."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16(workload: str, tensor: str, shape, scale: float, seed: int = 0) -> np.ndarray:
    """bf16 bits of ``N(0,1) * scale`` with the given shape, seeded per (workload, tensor)."""
    n = int(np.prod(shape)) if len(shape) else 1
    x = normal_f64(tensor_key(workload, tensor, seed), n) * scale
    return f32_to_bf16_bits(x.astype(np.float32)).reshape(shape)


BF16_NAN = np.uint16(0x7FC0)


def uint4_codes(workload: str, tensor: str, shape, seed: int = 0) -> np.ndarray:
    """4-bit codes (0..15, uint8) of the given shape: the low four bits of the stream's outputs."""
    n = int(np.prod(shape)) if len(shape) else 1
    return (splitmix64_stream(tensor_key(workload, tensor, seed), 0, n) & np.uint64(15)).astype(np.uint8).reshape(shape)


def uint32_words(workload: str, tensor: str, shape, seed: int = 0) -> np.ndarray:
    """Uniform 32-bit words (uint32) of the given shape: the low half of the stream's outputs.
    Read as eight 4-bit fields each, they are eight independent uniform codes."""
    n = int(np.prod(shape)) if len(shape) else 1
    return (splitmix64_stream(tensor_key(workload, tensor, seed), 0, n) & np.uint64(0xFFFFFFFF)).astype(
        np.uint32).reshape(shape)
