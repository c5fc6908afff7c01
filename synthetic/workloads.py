"""The five synthetic attention workloads and their seeded inputs.

Shapes follow the three stage signatures of the paper (Section 4, Table 1): a
prefill over a prompt, a prefill_kv of a new chunk over a history cache, and a
decode of one token per sequence over a length-masked static cache.  Values are
N(0,1)/sqrt(head_dim) rounded to bf16 (see ``gen``); the history part of a cache
is drawn the same way (history is arbitrary data).  Nothing here computes any
part of the attention method.

Layouts (all bf16 bit patterns, uint16):
  q    [B, S, Hq,  D]     token-major, as a q projection produces it
  k, v [B, S, Hkv, D]
  k_cache, v_cache [B, Hkv, L, D]   static maximum length L
  hist_len [B] int32 (decode only): valid history tokens of each sequence
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

from . import gen


@dataclasses.dataclass(frozen=True)
class Shape:
    name: str
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    max_len: int
    rope_theta: float

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.head_dim)


# Tiny 1-layer GQA attention; the stage chain prefill(16) -> prefill_kv(8 over 16) -> 4 decodes.
TINY = Shape("tiny", 1, 4, 2, 64, 32, 1.0e4)
# 7B-class prefill over a fully valid 512-token prompt.
PREFILL_7B = Shape("prefill_7b", 1, 28, 4, 128, 512, 1.0e6)
# 512-token chunk over 1536 history tokens, static max 2048.
PREFILL_KV = Shape("prefill_kv", 1, 32, 8, 128, 2048, 5.0e5)
# Decode sweep, static max 8192; batch and history length vary per point.
DECODE_BATCHES = (1, 4, 16)
DECODE_HISTS = (1024, 4096, 8191)


def decode_shape(batch: int) -> Shape:
    return Shape(f"decode_b{batch}", batch, 32, 8, 128, 8192, 5.0e5)


# Long context: prefill 4096; prefill_kv 4096 over 28672; decode at 32767 valid tokens.
LONG = Shape("long", 1, 40, 8, 128, 32768, 1.0e6)
LONG_PREFILL = 4096
LONG_PKV_HIST = 28672
LONG_PKV_CHUNK = 4096
LONG_DECODE_HIST = 32767


def tokens(shape: Shape, tag: str, n_tokens: int, seed: int = 0):
    """q, k, v for ``n_tokens`` new tokens of every sequence, drawn under stream tag ``tag``."""
    b, hq, hkv, d = shape.batch, shape.n_q_heads, shape.n_kv_heads, shape.head_dim
    s = shape.scale
    q = gen.normal_bf16(shape.name, f"{tag}/q", (b, n_tokens, hq, d), s, seed)
    k = gen.normal_bf16(shape.name, f"{tag}/k", (b, n_tokens, hkv, d), s, seed)
    v = gen.normal_bf16(shape.name, f"{tag}/v", (b, n_tokens, hkv, d), s, seed)
    return q, k, v


def cache(shape: Shape, tag: str, n_hist: int, fill: str = "zero", seed: int = 0):
    """k_cache, v_cache of shape [B, Hkv, L, D] with slots [0, n_hist) drawn at random.

    Slots ``>= n_hist`` hold ``fill``: "zero", "nan" (bf16 quiet NaN, to prove the
    stages never read them) or "random" (drawn from a separate stream).
    """
    b, hkv, L, d = shape.batch, shape.n_kv_heads, shape.max_len, shape.head_dim
    assert 0 <= n_hist <= L
    out = []
    for name in ("k_cache", "v_cache"):
        c = np.zeros((b, hkv, L, d), dtype=np.uint16)
        if fill == "nan":
            c[...] = gen.BF16_NAN
        elif fill == "random":
            c[...] = gen.normal_bf16(shape.name, f"{tag}/{name}/pad", (b, hkv, L, d), shape.scale, seed)
        elif fill != "zero":
            raise ValueError(fill)
        if n_hist:
            c[:, :, :n_hist, :] = gen.normal_bf16(shape.name, f"{tag}/{name}", (b, hkv, n_hist, d),
                                                  shape.scale, seed)
        out.append(c)
    return out[0], out[1]


def new_q_kv_are_views_of(shape: Shape, q, k, v, start: int, count: int):
    """Slice ``count`` tokens starting at token ``start`` (copies, contiguous)."""
    sl = slice(start, start + count)
    return (np.ascontiguousarray(q[:, sl]), np.ascontiguousarray(k[:, sl]),
            np.ascontiguousarray(v[:, sl]))
