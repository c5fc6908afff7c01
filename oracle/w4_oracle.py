"""CPU oracle of the W4BF16 weight-only GEMV -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the bench's CPU-baseline leg use it.

The paper deploys every model with W4BF16 quantization: 4-bit weights, bf16
activations (Section 5.1), and its decode throughput is set by streaming those
weights (Section 5.2).  The paper fixes no group size, zero-point convention or
storage layout; the reading taken here is the common grouped asymmetric form
(GPTQ/AWQ style): weight row n, input index k, group g = k // 128 along k, code
q[n,k] in 0..15, zero point z[n,g] in 0..15 and bf16 scale s[n,g]:

    W[n,k] = (q[n,k] - z[n,g]) * s[n,g]
    y[m,n] = sum_k x[m,k] * W[n,k]

computed here exactly in float64 from the bf16 inputs (``gemv``).

Storage written by ``write_tiles`` and read by ``unpack_tiles`` (this module's own writer and
reader of the documented format):
the matrix is cut into tiles of 16 rows x 128 inputs; tile (T, G) -- rows 16T..16T+15,
group G -- is the (T * K/128 + G)-th record of 1072 bytes:
  bytes    0..1023  codes: row r of the tile holds 16 little-endian uint32 words at
                    byte 64 r; word i carries k = 128 G + 8 i + j (j = 0..7) with the
                    nibble of j at bit offset (0, 16, 4, 20, 8, 24, 12, 28)[j]
  bytes 1024..1055  the 16 rows' scales, bf16 bits, row r at byte 1024 + 2 r
  bytes 1056..1071  the 16 rows' zero points, one byte each, row r at byte 1056 + r
Rows past N in the last row-tile are padding and ignored.

No arithmetic in this module is pinned by a value the paper prints: the paper gives
no worked example of the quantized product or of the block around attention.  The pins
are the definitions' own closed forms and brute force (tests/test_w4_oracle.py).
"""
from __future__ import annotations

import numpy as np

GROUP = 128
TILE_ROWS = 16
TILE_BYTES = 1072
CODE_BYTES = 1024
SCALE_OFFSET = 1024
ZERO_OFFSET = 1056
NIBBLE_SHIFT = (0, 16, 4, 20, 8, 24, 12, 28)


def unpack_row_words(words: np.ndarray) -> np.ndarray:
    """uint32 [..., K/8] -> codes uint8 [..., K] (the nibble order within a word)."""
    w = np.asarray(words, dtype=np.uint32)
    out = np.empty(w.shape[:-1] + (w.shape[-1] * 8,), dtype=np.uint8)
    for j, sh in enumerate(NIBBLE_SHIFT):
        out[..., j::8] = ((w >> np.uint32(sh)) & np.uint32(15)).astype(np.uint8)
    return out


def unpack_tiles(buf: np.ndarray, N: int, K: int):
    """Tile stream (uint8, ceil(N/16) * K/128 * 1072 bytes) -> (codes uint8 [N, K],
    scales bf16 bits uint16 [N, K/128], zeros uint8 [N, K/128])."""
    ng, nt = K // GROUP, (N + TILE_ROWS - 1) // TILE_ROWS
    b = np.asarray(buf, dtype=np.uint8)
    assert b.size == nt * ng * TILE_BYTES
    rec = b.reshape(nt, ng, TILE_BYTES)
    words = rec[:, :, :CODE_BYTES].copy().view("<u4").reshape(nt, ng, TILE_ROWS, 16)
    # [tile, group, row, word] -> [tile, row, group, word] -> rows x (K/8) words
    words = words.transpose(0, 2, 1, 3).reshape(nt * TILE_ROWS, ng * 16)
    scales = rec[:, :, SCALE_OFFSET:ZERO_OFFSET].copy().view("<u2").reshape(nt, ng, TILE_ROWS)
    zeros = rec[:, :, ZERO_OFFSET:TILE_BYTES].reshape(nt, ng, TILE_ROWS)
    scales = scales.transpose(0, 2, 1).reshape(nt * TILE_ROWS, ng)
    zeros = zeros.transpose(0, 2, 1).reshape(nt * TILE_ROWS, ng)
    return unpack_row_words(words)[:N], scales[:N].copy(), zeros[:N].copy()


def write_tiles(codes, scales_bf16, zeros) -> np.ndarray:
    """codes uint8 [N, K], scales bf16 bits uint16 [N, K/128], zeros uint8 [N, K/128] -> the
    tile stream (uint8, ceil(N/16) * K/128 * 1072 bytes), every value placed at the byte the
    format above names; padding rows of the last row-tile stay zero."""
    codes = np.asarray(codes, dtype=np.uint8)
    N, K = codes.shape
    ng, nt = K // GROUP, (N + TILE_ROWS - 1) // TILE_ROWS
    assert K % GROUP == 0 and np.shape(scales_bf16) == (N, ng) and np.shape(zeros) == (N, ng)
    buf = np.zeros(nt * ng * TILE_BYTES, dtype=np.uint8)
    n = np.arange(N)[:, None]
    k = np.arange(K)[None, :]
    rec = (n // TILE_ROWS) * ng + k // GROUP                      # record of (n, k)
    bit = np.asarray(NIBBLE_SHIFT)[k % 8]                          # bit of the code in its word
    byte = rec * TILE_BYTES + 64 * (n % TILE_ROWS) + 4 * ((k % GROUP) // 8) + bit // 8
    np.bitwise_or.at(buf, byte.ravel(), ((codes & 15) << (bit % 8)).astype(np.uint8).ravel())
    g = np.arange(ng)[None, :]
    rec = (n // TILE_ROWS) * ng + g                                # record of (n, group)
    s = np.asarray(scales_bf16, dtype=np.uint16)
    at = rec * TILE_BYTES + SCALE_OFFSET + 2 * (n % TILE_ROWS)
    buf[at.ravel()] = (s & 0xFF).astype(np.uint8).ravel()          # little-endian bf16 bits
    buf[(at + 1).ravel()] = (s >> 8).astype(np.uint8).ravel()
    buf[(rec * TILE_BYTES + ZERO_OFFSET + n % TILE_ROWS).ravel()] = np.asarray(zeros, np.uint8).ravel()
    return buf


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def dequant(codes, scales_bf16, zeros) -> np.ndarray:
    """W [N, K] float64 = (q - z) * s, groups of 128 along k."""
    q = np.asarray(codes, dtype=np.float64)
    z = np.repeat(np.asarray(zeros, dtype=np.float64), GROUP, axis=-1)
    s = np.repeat(bf16_to_f64(scales_bf16), GROUP, axis=-1)
    return (q - z) * s


def gemv(codes, scales_bf16, zeros, x_bf16) -> np.ndarray:
    """y [M, N] float64 = x [M, K] . W[N, K]^T, exactly in float64."""
    return bf16_to_f64(x_bf16) @ dequant(codes, scales_bf16, zeros).T


# ----------------------------------------------------------------------------- the block around attention
# Listing 1's attention half of a decoder block, for one decode step with W4BF16 weights:
#   xn = RMSNorm(x) * gamma                    (input_layernorm)
#   q | k | v = xn . Wqkv^T                    (q_proj, k_proj, v_proj stacked by rows)
#   o = attention(RoPE(q), RoPE(k) -> cache, v -> cache)   (the decode stage)
#   h = x + o . Wo^T                           (o_proj + residual)
# Readings (the paper gives the dataflow only): RMSNorm r = 1 / sqrt(mean(x^2) + eps) per row
# and x * r * gamma rounded once to bf16; q, k, v and o are bf16 (the stage's inputs and
# output); the residual is added before h is rounded to bf16.


def to_bf16_bits(v) -> np.ndarray:
    """float64 -> bf16 bits, round to nearest, ties to even (finite values in the normal range)."""
    a = np.asarray(v, dtype=np.float64)
    assert np.isfinite(a).all()
    m, e = np.frexp(a)                     # a = m * 2^e, 0.5 <= |m| < 1
    r = np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)  # 8 significant bits, ties to even
    return (r.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def rmsnorm(x_bf16, gamma_bf16, eps: float) -> np.ndarray:
    """bf16 bits [M, K] -> bf16 bits of x * r * gamma, r = 1 / sqrt(mean_k x^2 + eps) per row."""
    x = bf16_to_f64(x_bf16)
    r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    return to_bf16_bits(x * r * bf16_to_f64(gamma_bf16))


def decode_layer(shape, x_bf16, gamma_bf16, eps, wqkv, wo, hist, k_cache, v_cache, attn_oracle=None):
    """h (bf16 bits [B, hidden]) of one decode step; wqkv / wo are (codes, scales, zeros) of the
    stacked [(Hq + 2 Hkv) D, hidden] and the [hidden, Hq D] matrices.  The caches get the new k
    (rotated) and v at slot hist[b], as the decode stage does."""
    if attn_oracle is None:
        from oracle import oracle as attn_oracle
    B, D = shape.batch, shape.head_dim
    qd, kd = shape.n_q_heads * D, shape.n_kv_heads * D
    xn = rmsnorm(x_bf16, gamma_bf16, eps)
    qkv = to_bf16_bits(gemv(*wqkv, xn))
    q = qkv[:, :qd].reshape(B, 1, shape.n_q_heads, D)
    k = qkv[:, qd:qd + kd].reshape(B, 1, shape.n_kv_heads, D)
    v = qkv[:, qd + kd:].reshape(B, 1, shape.n_kv_heads, D)
    o = attn_oracle.decode(shape, q, k, v, hist, k_cache, v_cache).reshape(B, qd)
    return to_bf16_bits(bf16_to_f64(x_bf16) + gemv(*wo, o))


# ----------------------------------------------------------------------------- prefill-side GEMM
# For a chunk of T tokens the projections are GEMMs; their kernel decodes each weight into the
# tensor cores' bf16 operand, so the reading there is the usual dequantize-then-multiply one:
#   W_bf16[n, k] = bf16((q[n, k] - z[n, g]) * s[n, g])   (one rounding of each weight)
#   Y[t, n] = sum_k x[t, k] * W_bf16[n, k]               (exact here in float64)


def dequant_bf16(codes, scales_bf16, zeros) -> np.ndarray:
    """bf16 bits [N, K] of (q - z) * s, each rounded once to bf16."""
    return to_bf16_bits(dequant(codes, scales_bf16, zeros))


def gemm_bf16w(codes, scales_bf16, zeros, x_bf16) -> np.ndarray:
    """Y [T, N] float64 = x [T, K] . W_bf16[N, K]^T."""
    return bf16_to_f64(x_bf16) @ bf16_to_f64(dequant_bf16(codes, scales_bf16, zeros)).T


# ----------------------------------------------------------------------------- the block around attention, prefill
# Listing 1 for a prefill (hist = 0, Section 4.2) or prefill_kv (hist > 0, Section 4.3) chunk
# of S tokens per sequence, with the prefill-side projections (weights rounded once to bf16):
#   xn = RMSNorm(x) * gamma               per token
#   q | k | v = xn . Wqkv_bf16^T          rounded to bf16
#   o = attention of the chunk over its history (RoPE, cache append, causal mask)
#   h = x + o . Wo_bf16^T                 rounded to bf16


def prefill_layer(shape, x_bf16, gamma_bf16, eps, wqkv, wo, hist, k_cache, v_cache, attn_oracle=None):
    """h (bf16 bits [B, S, hidden]) of one chunk of S tokens per sequence over `hist`
    history tokens (the same for every sequence); x is [B, S, hidden].  The caches get the
    chunk's rotated k and its v at slots hist .. hist + S - 1, as the prefill stages do."""
    if attn_oracle is None:
        from oracle import oracle as attn_oracle
    B, S, hidden = np.shape(x_bf16)
    D = shape.head_dim
    qd, kd = shape.n_q_heads * D, shape.n_kv_heads * D
    x2 = np.asarray(x_bf16, dtype=np.uint16).reshape(B * S, hidden)
    xn = rmsnorm(x2, gamma_bf16, eps)
    qkv = to_bf16_bits(gemm_bf16w(*wqkv, xn))
    q = qkv[:, :qd].reshape(B, S, shape.n_q_heads, D).copy()
    k = qkv[:, qd:qd + kd].reshape(B, S, shape.n_kv_heads, D).copy()
    v = qkv[:, qd + kd:].reshape(B, S, shape.n_kv_heads, D).copy()
    o = attn_oracle.prefill_kv(shape, q, k, v, int(hist), k_cache, v_cache).reshape(B * S, qd)
    return to_bf16_bits(bf16_to_f64(x2) + gemm_bf16w(*wo, o)).reshape(B, S, hidden)
