"""W4BF16 weight-only GEMV through the C ABI (attn_w4bf16_gemv): packing and marshalling.

Weights of an [N, K] matrix: 4-bit codes q (0..15), per group of 128 inputs along k a
zero point z (0..15) and a bf16 scale s; W[n,k] = (q - z) * s and y = x . W^T.

The kernel reads one contiguous stream of tiles, each 16 rows x 128 inputs (one group)
with its own scales and zero points, so that every copy it issues is one contiguous
1072-byte record.  Tile (T, G) is record T * (K/128) + G:
  bytes    0..1023  codes, row r of the tile at byte 64 r as 16 uint32 words; word i
                    holds inputs 128 G + 8 i + j, the code of j at bit
                    (0, 16, 4, 20, 8, 24, 12, 28)[j] (the codes of k and k + 1 sit in
                    the two 16-bit halves, so one masked OR makes a bf16 pair of them)
  bytes 1024..1055  scales of rows 0..15 (bf16 bits)
  bytes 1056..1071  zero points of rows 0..15
The last row-tile is padded with zero codes, scales and zero points up to 16 rows.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _lib
from .attention import _stream

NIBBLE_SHIFT = (0, 16, 4, 20, 8, 24, 12, 28)
TILE_ROWS, TILE_BYTES = 16, 1072


def pack_codes(codes: np.ndarray) -> np.ndarray:
    """codes uint8 [N, K] (values 0..15, K a multiple of 8) -> row words uint32 [N, K / 8]."""
    c = np.asarray(codes, dtype=np.uint32)
    if c.shape[-1] % 8:
        raise ValueError("K must be a multiple of 8")
    words = np.zeros(c.shape[:-1] + (c.shape[-1] // 8,), dtype=np.uint32)
    for j, sh in enumerate(NIBBLE_SHIFT):
        words |= (c[..., j::8] & np.uint32(15)) << np.uint32(sh)
    return words


def pack_tiles(words: np.ndarray, scales: np.ndarray, zeros: np.ndarray) -> np.ndarray:
    """Row words uint32 [N, K/8], scales bf16 bits uint16 [N, K/128], zero points uint8
    [N, K/128] -> the tile stream (uint8, ceil(N/16) * (K/128) * 1072 bytes)."""
    words = np.asarray(words, dtype=np.uint32)
    N, kw = words.shape
    K = kw * 8
    if K % 128 or scales.shape != (N, K // 128) or zeros.shape != (N, K // 128):
        raise ValueError("shapes: words [N, K/8], scales and zeros [N, K/128], K a multiple of 128")
    ng, nt = K // 128, (N + TILE_ROWS - 1) // TILE_ROWS
    rows = nt * TILE_ROWS
    out = np.zeros((nt, ng, TILE_BYTES), dtype=np.uint8)
    w = np.zeros((rows, kw), dtype="<u4")
    w[:N] = words
    # rows x (groups x 16 words) -> [tile, group, row in tile, word]
    out[:, :, :1024] = w.reshape(nt, TILE_ROWS, ng, 16).transpose(0, 2, 1, 3).copy().view(np.uint8) \
        .reshape(nt, ng, 1024)
    s = np.zeros((rows, ng), dtype="<u2")
    s[:N] = scales
    out[:, :, 1024:1056] = s.reshape(nt, TILE_ROWS, ng).transpose(0, 2, 1).copy().view(np.uint8) \
        .reshape(nt, ng, 32)
    z = np.zeros((rows, ng), dtype=np.uint8)
    z[:N] = zeros
    out[:, :, 1056:] = z.reshape(nt, TILE_ROWS, ng).transpose(0, 2, 1)
    return out.reshape(-1)


def w4bf16_gemv(tiles: torch.Tensor, x: torch.Tensor, N: int, out=None, stream=None, err=None,
                weights_static: bool = False) -> torch.Tensor:
    """y [M, N] (bf16) = x [M, K] . W^T for the tile stream of an [N, K] matrix (a uint8
    CUDA tensor from pack_tiles) and x bf16 [M, K] on the same device.  err: optional
    int32 CUDA tensor whose bit ATTN_DEVERR_TIMEOUT the kernel sets when a wait runs out.
    weights_static: the kernel right before this call on the stream does not write the
    tiles, so the call may start streaming them before that kernel has finished."""
    lib = _lib.load()
    M, K = x.shape
    for t, name in ((tiles, "tiles"), (x, "x")):
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()):
            raise TypeError(f"{name} must be a contiguous CUDA tensor")
    if x.dtype != torch.bfloat16 or tiles.dtype != torch.uint8:
        raise TypeError("dtypes: tiles uint8, x bf16")
    if K % 128 or tiles.numel() != (N + TILE_ROWS - 1) // TILE_ROWS * (K // 128) * TILE_BYTES:
        raise ValueError("tiles must hold ceil(N/16) * (K/128) records of 1072 bytes, K a multiple of 128")
    if out is None:
        out = torch.empty((M, N), dtype=x.dtype, device=x.device)
    elif out.dtype != torch.bfloat16 or tuple(out.shape) != (M, N) or not out.is_contiguous() or not out.is_cuda:
        raise ValueError("out must be a contiguous CUDA bf16 tensor [M, N]")
    if err is not None and not (isinstance(err, torch.Tensor) and err.is_cuda and err.dtype == torch.int32):
        raise TypeError("err must be an int32 CUDA tensor")
    rc = lib.attn_w4bf16_gemv(tiles.data_ptr(), x.data_ptr(), M, N, K, out.data_ptr(),
                              None if err is None else err.data_ptr(),
                              _lib.W4_WEIGHTS_STATIC if weights_static else 0, _stream(stream))
    if rc != _lib.ATTN_OK:
        raise _lib.AttnError(rc, "attn_w4bf16_gemv", lib)
    return out


def w4bf16_gemv_fused(tiles: torch.Tensor, x: torch.Tensor, N: int, rms_gamma=None, rms_eps: float = 0.0,
                      residual=None, out=None, split=None, stream=None, err=None,
                      weights_static: bool = False):
    """w4bf16_gemv with the fused parts of attn_w4bf16_gemv_fused: RMSNorm of x by rms_gamma
    (bf16 [K]), a residual (bf16 [M, N]) added before rounding, and split = (n0, n1) to return
    the output columns as three tensors [M, n0], [M, n1 - n0], [M, N - n1]."""
    lib = _lib.load()
    M, K = x.shape
    for t, name in ((tiles, "tiles"), (x, "x")):
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()):
            raise TypeError(f"{name} must be a contiguous CUDA tensor")
    if x.dtype != torch.bfloat16 or tiles.dtype != torch.uint8:
        raise TypeError("dtypes: tiles uint8, x bf16")
    if K % 128 or tiles.numel() != (N + TILE_ROWS - 1) // TILE_ROWS * (K // 128) * TILE_BYTES:
        raise ValueError("tiles must hold ceil(N/16) * (K/128) records of 1072 bytes, K a multiple of 128")
    for t, name, shape in ((rms_gamma, "rms_gamma", (K,)), (residual, "residual", (M, N))):
        if t is not None and not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()
                                  and t.dtype == torch.bfloat16 and tuple(t.shape) == shape):
            raise TypeError(f"{name} must be a contiguous CUDA bf16 tensor of shape {shape}")
    if split is None:
        outs = [torch.empty((M, N), dtype=x.dtype, device=x.device) if out is None else out]
        n0 = n1 = 0
    else:
        n0, n1 = split
        outs = [torch.empty((M, w), dtype=x.dtype, device=x.device) for w in (n0, n1 - n0, N - n1)]
    if err is not None and not (isinstance(err, torch.Tensor) and err.is_cuda and err.dtype == torch.int32):
        raise TypeError("err must be an int32 CUDA tensor")
    ptr = (lambda t: None if t is None else t.data_ptr())
    rc = lib.attn_w4bf16_gemv_fused(tiles.data_ptr(), x.data_ptr(), M, N, K, ptr(rms_gamma), float(rms_eps),
                                    ptr(residual), outs[0].data_ptr(), n0, ptr(outs[1]) if split else None, n1,
                                    ptr(outs[2]) if split else None, ptr(err),
                                    _lib.W4_WEIGHTS_STATIC if weights_static else 0, _stream(stream))
    if rc != _lib.ATTN_OK:
        raise _lib.AttnError(rc, "attn_w4bf16_gemv_fused", lib)
    return outs[0] if split is None else tuple(outs)


def w4bf16_gemm(tiles: torch.Tensor, x: torch.Tensor, N: int, out=None, stream=None, err=None) -> torch.Tensor:
    """Y [T, N] (bf16) = x [T, K] . W_bf16^T on the tensor cores (attn_w4bf16_gemm), for a chunk of
    T tokens; W_bf16 = bf16((q - z) s) from the tile stream of an [N, K] matrix."""
    lib = _lib.load()
    T, K = x.shape
    for t, name in ((tiles, "tiles"), (x, "x")):
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()):
            raise TypeError(f"{name} must be a contiguous CUDA tensor")
    if x.dtype != torch.bfloat16 or tiles.dtype != torch.uint8:
        raise TypeError("dtypes: tiles uint8, x bf16")
    if K % 128 or N % 128 or tiles.numel() != N // TILE_ROWS * (K // 128) * TILE_BYTES:
        raise ValueError("N and K multiples of 128; tiles must hold N/16 * K/128 records of 1072 bytes")
    if out is None:
        out = torch.empty((T, N), dtype=x.dtype, device=x.device)
    elif out.dtype != torch.bfloat16 or tuple(out.shape) != (T, N) or not out.is_contiguous() or not out.is_cuda:
        raise ValueError("out must be a contiguous CUDA bf16 tensor [T, N]")
    if err is not None and not (isinstance(err, torch.Tensor) and err.is_cuda and err.dtype == torch.int32):
        raise TypeError("err must be an int32 CUDA tensor")
    rc = lib.attn_w4bf16_gemm(tiles.data_ptr(), x.data_ptr(), T, N, K, out.data_ptr(),
                              None if err is None else err.data_ptr(), _stream(stream))
    if rc != _lib.ATTN_OK:
        raise _lib.AttnError(rc, "attn_w4bf16_gemm", lib)
    return out
