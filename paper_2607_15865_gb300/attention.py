"""Torch-facing wrapper of the C ABI: one context per attention shape.

Argument marshalling only -- every stage runs in the library's CUDA kernels:

  prefill     (Section 4.2)  q [B,S,Hq,D], k/v [B,S,Hkv,D] at positions 0..S-1
  prefill_kv  (Section 4.3)  the same at positions hist..hist+S-1 over hist cached tokens
  decode      (Section 4.4)  q [B,1,Hq,D], k/v [B,1,Hkv,D], hist_len [B] int32 on the device
              (decode_multi: q [B,n,Hq,D], k/v [B,n,Hkv,D], n new tokens per sequence)

and the stage driver of Sections 4.1 and 4.5:

  prompt        a prompt of any length in segments: 1 prefill (or prefill_kv) + N prefill_kv
  decode_steps  n decode steps in a row, step t at positions hist_len + t (step-major inputs)

Caches are [B,Hkv,L,D] bf16 tensors owned by the caller and updated in place.
All calls are asynchronous on the given (default: current) torch CUDA stream.
"""
from __future__ import annotations

import ctypes

import torch

from . import _lib

_BF16_LIKE = (torch.bfloat16, torch.int16, torch.uint16)


def _ptr(t: torch.Tensor, name: str, shape=None) -> int:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype not in _BF16_LIKE:
        raise TypeError(f"{name} must hold bf16 values (torch.bfloat16 or 16-bit integer bit patterns)")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t.data_ptr()


def _stream(stream) -> int:
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


class Attention:
    """A context of include/attn.h for one (batch, heads, head_dim, max_len, theta) shape."""

    def __init__(self, batch: int, n_q_heads: int, n_kv_heads: int, head_dim: int, max_len: int,
                 rope_theta: float):
        self.lib = _lib.load()
        self.batch, self.n_q_heads, self.n_kv_heads = batch, n_q_heads, n_kv_heads
        self.head_dim, self.max_len, self.rope_theta = head_dim, max_len, float(rope_theta)
        cfg = _lib.AttnCfg(batch, n_q_heads, n_kv_heads, head_dim, max_len, float(rope_theta))
        handle = ctypes.c_void_p()
        rc = self.lib.attn_create(ctypes.byref(cfg), ctypes.byref(handle))
        if rc != _lib.ATTN_OK:
            raise _lib.AttnError(rc, "attn_create", self.lib)
        self._ctx = handle

    @classmethod
    def for_shape(cls, shape) -> "Attention":
        return cls(shape.batch, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.max_len, shape.rope_theta)

    @property
    def handle(self) -> ctypes.c_void_p:
        return self._ctx

    def close(self):
        if getattr(self, "_ctx", None) is not None and self._ctx.value:
            self.lib.attn_destroy(self._ctx)
            self._ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, rc: int, what: str):
        if rc != _lib.ATTN_OK:
            raise _lib.AttnError(rc, what, self.lib)

    def _cache_shape(self):
        return (self.batch, self.n_kv_heads, self.max_len, self.head_dim)

    def _new_out(self, q: torch.Tensor, out):
        return torch.empty_like(q) if out is None else out

    def prefill(self, q, k, v, k_cache, v_cache, out=None, stream=None) -> torch.Tensor:
        return self.prefill_kv(q, k, v, 0, k_cache, v_cache, out, stream, _stage="attn_prefill")

    def prefill_kv(self, q, k, v, hist_len: int, k_cache, v_cache, out=None, stream=None,
                   _stage: str = "attn_prefill_kv") -> torch.Tensor:
        B, S = q.shape[0], q.shape[1]
        qs = (self.batch, S, self.n_q_heads, self.head_dim)
        ks = (self.batch, S, self.n_kv_heads, self.head_dim)
        out = self._new_out(q, out)
        args = (_ptr(q, "q", qs), _ptr(k, "k", ks), _ptr(v, "v", ks))
        cache = (_ptr(k_cache, "k_cache", self._cache_shape()), _ptr(v_cache, "v_cache", self._cache_shape()),
                 _ptr(out, "out", qs))
        if _stage == "attn_prefill":
            rc = self.lib.attn_prefill(self._ctx, *args, S, *cache, _stream(stream))
        else:
            rc = self.lib.attn_prefill_kv(self._ctx, *args, int(hist_len), S, *cache, _stream(stream))
        self._check(rc, _stage)
        return out

    def decode(self, q, k, v, hist_len: torch.Tensor, k_cache, v_cache, out=None, stream=None) -> torch.Tensor:
        qs = (self.batch, 1, self.n_q_heads, self.head_dim)
        ks = (self.batch, 1, self.n_kv_heads, self.head_dim)
        if not (isinstance(hist_len, torch.Tensor) and hist_len.is_cuda and hist_len.dtype == torch.int32
                and hist_len.is_contiguous() and tuple(hist_len.shape) == (self.batch,)):
            raise TypeError("hist_len must be a contiguous int32 CUDA tensor of shape [batch]")
        out = self._new_out(q, out)
        rc = self.lib.attn_decode(self._ctx, _ptr(q, "q", qs), _ptr(k, "k", ks), _ptr(v, "v", ks),
                                  hist_len.data_ptr(), _ptr(k_cache, "k_cache", self._cache_shape()),
                                  _ptr(v_cache, "v_cache", self._cache_shape()), _ptr(out, "out", qs),
                                  _stream(stream))
        self._check(rc, "attn_decode")
        return out

    def decode_multi(self, q, k, v, hist_len: torch.Tensor, k_cache, v_cache, out=None,
                     stream=None) -> torch.Tensor:
        """n = q.shape[1] new tokens per sequence at positions hist_len[b] + i (causal among them)."""
        n = q.shape[1]
        qs = (self.batch, n, self.n_q_heads, self.head_dim)
        ks = (self.batch, n, self.n_kv_heads, self.head_dim)
        if not (isinstance(hist_len, torch.Tensor) and hist_len.is_cuda and hist_len.dtype == torch.int32
                and hist_len.is_contiguous() and tuple(hist_len.shape) == (self.batch,)):
            raise TypeError("hist_len must be a contiguous int32 CUDA tensor of shape [batch]")
        out = self._new_out(q, out)
        rc = self.lib.attn_decode_multi(self._ctx, _ptr(q, "q", qs), _ptr(k, "k", ks), _ptr(v, "v", ks),
                                        hist_len.data_ptr(), n, _ptr(k_cache, "k_cache", self._cache_shape()),
                                        _ptr(v_cache, "v_cache", self._cache_shape()), _ptr(out, "out", qs),
                                        _stream(stream))
        self._check(rc, "attn_decode_multi")
        return out

    def decode_layer(self, x, rms_gamma, rms_eps: float, wqkv_tiles, wo_tiles, hist_len: torch.Tensor, k_cache,
                     v_cache, out=None, weights_static: bool = False, stream=None) -> torch.Tensor:
        """One decode step of the attention half of a decoder block with W4BF16 weights
        (attn_decode_layer): x [B, hidden] -> x + o_proj(attention(qkv_proj(RMSNorm(x))))."""
        hidden = x.shape[-1]
        if not (isinstance(hist_len, torch.Tensor) and hist_len.is_cuda and hist_len.dtype == torch.int32
                and hist_len.is_contiguous() and tuple(hist_len.shape) == (self.batch,)):
            raise TypeError("hist_len must be a contiguous int32 CUDA tensor of shape [batch]")
        for t, name in ((wqkv_tiles, "wqkv_tiles"), (wo_tiles, "wo_tiles")):
            if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous() and t.dtype == torch.uint8):
                raise TypeError(f"{name} must be a contiguous uint8 CUDA tensor (a W4BF16 tile stream)")
        qd, kd = self.n_q_heads * self.head_dim, self.n_kv_heads * self.head_dim
        if wqkv_tiles.numel() != (qd + 2 * kd + 15) // 16 * (hidden // 128) * 1072 or \
                wo_tiles.numel() != (hidden + 15) // 16 * (qd // 128) * 1072:
            raise ValueError("tile streams must hold [(Hq + 2 Hkv) D, hidden] and [hidden, Hq D] matrices")
        xs = (self.batch, hidden)
        out = self._new_out(x, out)
        rc = self.lib.attn_decode_layer(self._ctx, _ptr(x, "x", xs), _ptr(rms_gamma, "rms_gamma", (hidden,)),
                                        float(rms_eps), wqkv_tiles.data_ptr(), wo_tiles.data_ptr(), hidden,
                                        hist_len.data_ptr(), _ptr(k_cache, "k_cache", self._cache_shape()),
                                        _ptr(v_cache, "v_cache", self._cache_shape()), _ptr(out, "out", xs),
                                        _lib.W4_WEIGHTS_STATIC if weights_static else 0, _stream(stream))
        self._check(rc, "attn_decode_layer")
        return out

    def prefill_layer(self, x, rms_gamma, rms_eps: float, wqkv_tiles, wo_tiles, hist_len: int, k_cache, v_cache,
                      out=None, workspace=None, stream=None) -> torch.Tensor:
        """The attention half of a decoder block over a prefill / prefill_kv chunk with W4BF16
        weights (attn_prefill_layer): x [B, S, hidden] -> x + o_proj(attention(qkv_proj(RMSNorm(x)))),
        the chunk at positions hist_len ..  workspace: a uint8 CUDA tensor of at least
        prefill_layer_workspace(hidden, S) bytes (allocated here when None)."""
        if x.dim() != 3 or x.shape[0] != self.batch:
            raise ValueError("x must be [batch, chunk_len, hidden]")
        S, hidden = x.shape[1], x.shape[2]
        for t, name in ((wqkv_tiles, "wqkv_tiles"), (wo_tiles, "wo_tiles")):
            if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous() and t.dtype == torch.uint8):
                raise TypeError(f"{name} must be a contiguous uint8 CUDA tensor (a W4BF16 tile stream)")
        qd, kd = self.n_q_heads * self.head_dim, self.n_kv_heads * self.head_dim
        if wqkv_tiles.numel() != (qd + 2 * kd + 15) // 16 * (hidden // 128) * 1072 or \
                wo_tiles.numel() != (hidden + 15) // 16 * (qd // 128) * 1072:
            raise ValueError("tile streams must hold [(Hq + 2 Hkv) D, hidden] and [hidden, Hq D] matrices")
        need = self.prefill_layer_workspace(hidden, S)
        if workspace is None:
            workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
        if not (isinstance(workspace, torch.Tensor) and workspace.is_cuda and workspace.dtype == torch.uint8
                and workspace.is_contiguous() and workspace.numel() >= need):
            raise TypeError(f"workspace must be a contiguous uint8 CUDA tensor of at least {need} bytes")
        xs = (self.batch, S, hidden)
        out = self._new_out(x, out)
        rc = self.lib.attn_prefill_layer(self._ctx, _ptr(x, "x", xs), _ptr(rms_gamma, "rms_gamma", (hidden,)),
                                         float(rms_eps), wqkv_tiles.data_ptr(), wo_tiles.data_ptr(), hidden,
                                         int(hist_len), S, _ptr(k_cache, "k_cache", self._cache_shape()),
                                         _ptr(v_cache, "v_cache", self._cache_shape()), _ptr(out, "out", xs),
                                         workspace.data_ptr(), workspace.numel(), _stream(stream))
        self._check(rc, "attn_prefill_layer")
        return out

    def prefill_layer_workspace(self, hidden: int, chunk_len: int) -> int:
        """Bytes of device workspace attn_prefill_layer needs (host only)."""
        return int(self.lib.attn_prefill_layer_workspace(self._ctx, int(hidden), int(chunk_len)))

    def prompt(self, q, k, v, hist_len: int, seg_len: int, k_cache, v_cache, out=None,
               stream=None) -> torch.Tensor:
        """The whole prompt q [B,P,Hq,D], k/v [B,P,Hkv,D] at positions hist_len.. in segments of seg_len."""
        P = q.shape[1]
        qs = (self.batch, P, self.n_q_heads, self.head_dim)
        ks = (self.batch, P, self.n_kv_heads, self.head_dim)
        out = self._new_out(q, out)
        rc = self.lib.attn_prompt(self._ctx, _ptr(q, "q", qs), _ptr(k, "k", ks), _ptr(v, "v", ks), int(hist_len), P,
                                  int(seg_len), _ptr(k_cache, "k_cache", self._cache_shape()),
                                  _ptr(v_cache, "v_cache", self._cache_shape()), _ptr(out, "out", qs),
                                  _stream(stream))
        self._check(rc, "attn_prompt")
        return out

    def decode_steps(self, q, k, v, hist_len: torch.Tensor, k_cache, v_cache, out=None,
                     stream=None) -> torch.Tensor:
        """n = q.shape[0] decode steps; q [n,B,1,Hq,D], k/v [n,B,1,Hkv,D]; step t at hist_len + t."""
        n = q.shape[0]
        qs = (n, self.batch, 1, self.n_q_heads, self.head_dim)
        ks = (n, self.batch, 1, self.n_kv_heads, self.head_dim)
        if not (isinstance(hist_len, torch.Tensor) and hist_len.is_cuda and hist_len.dtype == torch.int32
                and hist_len.is_contiguous() and tuple(hist_len.shape) == (self.batch,)):
            raise TypeError("hist_len must be a contiguous int32 CUDA tensor of shape [batch]")
        out = self._new_out(q, out)
        rc = self.lib.attn_decode_steps(self._ctx, _ptr(q, "q", qs), _ptr(k, "k", ks), _ptr(v, "v", ks),
                                        hist_len.data_ptr(), n, _ptr(k_cache, "k_cache", self._cache_shape()),
                                        _ptr(v_cache, "v_cache", self._cache_shape()), _ptr(out, "out", qs),
                                        _stream(stream))
        self._check(rc, "attn_decode_steps")
        return out

    def timing_enable(self, max_launches: int):
        """Record CUDA events around every kernel of the following calls (0 disables)."""
        self._check(self.lib.attn_timing_enable(self._ctx, int(max_launches)), "attn_timing_enable")

    def timing_read(self):
        """Synchronise; returns {kernel: (milliseconds, launches)} since the last read."""
        ms = (ctypes.c_double * 4)()
        n = (ctypes.c_longlong * 4)()
        self._check(self.lib.attn_timing_read(self._ctx, ms, n), "attn_timing_read")
        return {name: (ms[i], n[i]) for i, name in enumerate(_lib.KERNELS)}

    def set_wait_limit(self, limit_ns: int):
        """Time limit of the kernels' bounded waits for the following calls, in nanoseconds
        (<= 0 restores the default of 1 s); see attn_set_wait_limit."""
        self._check(self.lib.attn_set_wait_limit(self._ctx, int(limit_ns)), "attn_set_wait_limit")

    def device_error(self, stream=None) -> int:
        """Synchronise, read and clear the device error word; returns its DEVERR_* bits."""
        flags = ctypes.c_int(0)
        rc = self.lib.attn_device_error(self._ctx, _stream(stream), ctypes.byref(flags))
        if rc not in (_lib.ATTN_OK, _lib.ATTN_EDEVICE):
            raise _lib.AttnError(rc, "attn_device_error", self.lib)
        return flags.value
