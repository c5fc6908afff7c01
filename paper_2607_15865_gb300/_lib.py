"""ctypes binding of ``libattn_gb300.so`` (include/attn.h): argument marshalling only.

Every stage runs in the library's CUDA kernels; this module never computes any
part of it and has no fallback: if the library is missing or cannot be loaded it
raises.  Tensors are torch CUDA tensors (torch provides device memory and
streams); bf16 tensors may be torch.bfloat16 or int16/uint16 bit patterns.
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libattn_gb300.so")

ATTN_OK, ATTN_EINVAL, ATTN_EARCH, ATTN_ECUDA, ATTN_ENOMEM, ATTN_EDEVICE = 0, -1, -2, -3, -4, -5
W4_WEIGHTS_STATIC = 1
DEVERR_HIST_RANGE, DEVERR_TIMEOUT = 1, 2

EXPORTED = ("attn_create", "attn_destroy", "attn_prefill", "attn_prefill_kv", "attn_decode",
            "attn_decode_multi", "attn_prompt", "attn_decode_steps", "attn_device_error", "attn_set_wait_limit",
            "attn_timing_enable", "attn_timing_read",
            "attn_strerror", "attn_last_cuda_error_string", "attn_decode_noalloc", "attn_w4bf16_gemv",
            "attn_w4bf16_rows_per_launch", "attn_w4bf16_gemv_fused", "attn_decode_layer",
            "attn_w4bf16_gemm", "attn_prefill_layer", "attn_prefill_layer_workspace")
NOALLOC_SCRATCH_FLOATS = 1 << 20
KERNELS = ("rope_append", "flash_fwd", "decode_split", "decode_combine")


class AttnCfg(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("n_q_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("max_len", ctypes.c_int), ("rope_theta", ctypes.c_double)]


class AttnError(RuntimeError):
    def __init__(self, code: int, what: str, lib=None):
        msg = f"{what}: {code}"
        if lib is not None:
            msg += f" ({lib.attn_strerror(code).decode()})"
            if code == ATTN_ECUDA:
                msg += f": {lib.attn_last_cuda_error_string().decode()}"
        super().__init__(msg)
        self.code = code


_lib = None


def load(path: str = LIB_PATH):
    """Load the library (once) and declare its signatures.  Raises if it is absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with paper_2607_15865_gb300.build.build() "
                          "(or __graft_entry__.build()); there is no fallback path")
    lib = ctypes.CDLL(path)
    vp, i32, u16p = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p
    lib.attn_create.argtypes = [ctypes.POINTER(AttnCfg), ctypes.POINTER(ctypes.c_void_p)]
    lib.attn_create.restype = i32
    lib.attn_destroy.argtypes = [vp]
    lib.attn_destroy.restype = None
    lib.attn_prefill.argtypes = [vp, u16p, u16p, u16p, i32, u16p, u16p, u16p, vp]
    lib.attn_prefill.restype = i32
    lib.attn_prefill_kv.argtypes = [vp, u16p, u16p, u16p, i32, i32, u16p, u16p, u16p, vp]
    lib.attn_prefill_kv.restype = i32
    lib.attn_decode.argtypes = [vp, u16p, u16p, u16p, vp, u16p, u16p, u16p, vp]
    lib.attn_decode.restype = i32
    lib.attn_decode_multi.argtypes = [vp, u16p, u16p, u16p, vp, i32, u16p, u16p, u16p, vp]
    lib.attn_decode_multi.restype = i32
    lib.attn_prompt.argtypes = [vp, u16p, u16p, u16p, i32, i32, i32, u16p, u16p, u16p, vp]
    lib.attn_prompt.restype = i32
    lib.attn_decode_steps.argtypes = [vp, u16p, u16p, u16p, vp, i32, u16p, u16p, u16p, vp]
    lib.attn_decode_steps.restype = i32
    lib.attn_device_error.argtypes = [vp, vp, ctypes.POINTER(ctypes.c_int)]
    lib.attn_device_error.restype = i32
    lib.attn_set_wait_limit.argtypes = [vp, ctypes.c_longlong]
    lib.attn_set_wait_limit.restype = i32
    lib.attn_timing_enable.argtypes = [vp, i32]
    lib.attn_timing_enable.restype = i32
    lib.attn_timing_read.argtypes = [vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_longlong)]
    lib.attn_timing_read.restype = i32
    lib.attn_decode_noalloc.argtypes = [ctypes.POINTER(AttnCfg), vp, vp, u16p, u16p, u16p, vp, u16p, u16p, u16p,
                                        vp, vp]
    lib.attn_decode_noalloc.restype = i32
    lib.attn_w4bf16_gemv.argtypes = [vp, u16p, i32, i32, i32, u16p, vp, i32, vp]
    lib.attn_w4bf16_gemv.restype = i32
    lib.attn_w4bf16_gemv_fused.argtypes = [vp, u16p, i32, i32, i32, u16p, ctypes.c_float, u16p, u16p, i32, u16p, i32,
                                           u16p, vp, i32, vp]
    lib.attn_w4bf16_gemv_fused.restype = i32
    lib.attn_decode_layer.argtypes = [vp, u16p, u16p, ctypes.c_float, vp, vp, i32, vp, u16p, u16p, u16p, i32, vp]
    lib.attn_decode_layer.restype = i32
    lib.attn_prefill_layer.argtypes = [vp, u16p, u16p, ctypes.c_float, vp, vp, i32, i32, i32, u16p, u16p, u16p, vp,
                                       ctypes.c_size_t, vp]
    lib.attn_prefill_layer.restype = i32
    lib.attn_prefill_layer_workspace.argtypes = [vp, i32, i32]
    lib.attn_prefill_layer_workspace.restype = ctypes.c_size_t
    lib.attn_w4bf16_gemm.argtypes = [vp, u16p, i32, i32, i32, u16p, vp, vp]
    lib.attn_w4bf16_gemm.restype = i32
    lib.attn_w4bf16_rows_per_launch.argtypes = [i32]
    lib.attn_w4bf16_rows_per_launch.restype = i32
    lib.attn_strerror.argtypes = [i32]
    lib.attn_strerror.restype = ctypes.c_char_p
    lib.attn_last_cuda_error_string.argtypes = []
    lib.attn_last_cuda_error_string.restype = ctypes.c_char_p
    _lib = lib
    return lib
