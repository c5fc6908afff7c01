"""The C-ABI library builds, loads and exports every function include/attn.h declares.

No compute call is made (no GPU here): only the host-side argument checks, which
run before any CUDA call, and the error strings.
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2607_15865_gb300 import _lib, build
    build.build()
    return _lib.load()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "attn.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(attn_\w+)\s*\(", text)))


def test_header_declares_the_stage_entry_points():
    names = declared_functions()
    for n in ("attn_create", "attn_destroy", "attn_prefill", "attn_prefill_kv", "attn_decode"):
        assert n in names


def test_library_exports_every_declared_function(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in include/attn.h but not exported"


def test_binding_declares_every_exported_function():
    from paper_2607_15865_gb300 import _lib
    assert sorted(_lib.EXPORTED) == [n for n in declared_functions() if n in _lib.EXPORTED]
    assert set(declared_functions()) <= set(_lib.EXPORTED) | set()


@pytest.mark.parametrize("cfg", [
    (0, 4, 2, 128, 64, 1e4),      # batch 0
    (1, 6, 4, 128, 64, 1e4),      # Hq not a multiple of Hkv
    (1, 34, 2, 128, 64, 1e4),     # group size 17 > 16
    (1, 4, 2, 96, 64, 1e4),       # head_dim 96
    (1, 4, 2, 128, 0, 1e4),       # max_len 0
    (1, 4, 2, 128, 64, -1.0),     # theta <= 0
    (1, 4, 2, 128, 64, float("inf")),
])
def test_create_rejects_invalid_shapes_on_the_host(lib, cfg):
    from paper_2607_15865_gb300 import _lib
    c = _lib.AttnCfg(*cfg)
    h = ctypes.c_void_p(123)
    assert lib.attn_create(ctypes.byref(c), ctypes.byref(h)) == _lib.ATTN_EINVAL
    assert not h.value, "a rejected create must return a NULL context"


def test_stage_calls_reject_null_context(lib):
    from paper_2607_15865_gb300 import _lib
    nul = None
    assert lib.attn_prefill(nul, nul, nul, nul, 4, nul, nul, nul, nul) == _lib.ATTN_EINVAL
    assert lib.attn_prefill_kv(nul, nul, nul, nul, 0, 4, nul, nul, nul, nul) == _lib.ATTN_EINVAL
    assert lib.attn_decode(nul, nul, nul, nul, nul, nul, nul, nul, nul) == _lib.ATTN_EINVAL
    assert lib.attn_device_error(nul, nul, None) == _lib.ATTN_EINVAL
    lib.attn_destroy(nul)


def test_error_strings(lib):
    for code in (0, -1, -2, -3, -4, -5, -99):
        assert lib.attn_strerror(code)
    assert lib.attn_last_cuda_error_string() is not None
