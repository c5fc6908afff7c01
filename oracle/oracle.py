"""ctypes front end of the CPU oracle (``attn_oracle.c``) -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the bench's CPU-baseline /
reference leg import this module.  It builds ``liboracle_attn.so`` with gcc on
first use (``-ffp-contract=off`` so that x86-64 and aarch64 round the RoPE
products identically) and wraps each C entry point for numpy arrays of bf16 bit
patterns (uint16).  The functions follow the paper's stages (Section 4): see the
header comment of ``attn_oracle.c`` for the definition and the readings taken.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attn_oracle.c")
_LIB = os.path.join(_HERE, "liboracle_attn.so")
_lock = threading.Lock()
_lib = None


class OracleCfg(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("n_q_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("max_len", ctypes.c_int), ("rope_theta", ctypes.c_double)]


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle into a shared library (plain C11, -O2, no FMA contraction)."""
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
                        "-shared", "-o", tmp, src, "-lm"], check=True)
        os.replace(tmp, out)
    return out


_U16P = np.ctypeslib.ndpointer(dtype=np.uint16, flags="C_CONTIGUOUS")
_I32P = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_F32P = np.ctypeslib.ndpointer(dtype=np.float32, flags="C_CONTIGUOUS")


def _bind(lib):
    cp = ctypes.POINTER(OracleCfg)
    lib.oracle_rope_tables.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_double, _F32P, _F32P]
    lib.oracle_rope_row.argtypes = [ctypes.c_int, _F32P, _F32P, _U16P, _F32P]
    lib.oracle_rope_row.restype = None
    lib.oracle_append.argtypes = [cp, _U16P, _U16P, _I32P, ctypes.c_int, ctypes.c_int, _U16P, _U16P]
    lib.oracle_attend.argtypes = [cp, _U16P, _I32P, ctypes.c_int, ctypes.c_int, _U16P, _U16P, _U16P,
                                  ctypes.c_int, ctypes.c_void_p]
    lib.oracle_prefill.argtypes = [cp, _U16P, _U16P, _U16P, ctypes.c_int, _U16P, _U16P, _U16P]
    lib.oracle_prefill_kv.argtypes = [cp, _U16P, _U16P, _U16P, ctypes.c_int, ctypes.c_int, _U16P, _U16P,
                                      _U16P]
    lib.oracle_decode.argtypes = [cp, _U16P, _U16P, _U16P, _I32P, _U16P, _U16P, _U16P]
    for f in (lib.oracle_rope_tables, lib.oracle_append, lib.oracle_attend, lib.oracle_prefill,
              lib.oracle_prefill_kv, lib.oracle_decode):
        f.restype = ctypes.c_int
    return lib


def load(path: str | None = None):
    """Load (building if needed) the oracle library; ``path`` loads another build of it."""
    global _lib
    if path is not None:
        return _bind(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
    return _lib


class OracleError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != 0:
        raise OracleError(f"oracle {what} rejected its arguments (rc={rc})")


def cfg_of(shape) -> OracleCfg:
    return OracleCfg(shape.batch, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.max_len,
                     float(shape.rope_theta))


def _u16(a):
    a = np.ascontiguousarray(a)
    assert a.dtype == np.uint16, a.dtype
    return a


def rope_tables(max_len: int, head_dim: int, theta: float, lib=None):
    lib = lib or load()
    c = np.empty((max_len, head_dim // 2), np.float32)
    s = np.empty_like(c)
    _check(lib.oracle_rope_tables(max_len, head_dim, float(theta), c, s), "rope_tables")
    return c, s


def rope_row(x_bf16, cos_row, sin_row, lib=None):
    lib = lib or load()
    x = _u16(x_bf16)
    y = np.empty(x.shape[-1], np.float32)
    lib.oracle_rope_row(x.shape[-1], np.ascontiguousarray(cos_row, np.float32),
                        np.ascontiguousarray(sin_row, np.float32), x, y)
    return y


def prefill(shape, q, k, v, k_cache, v_cache, lib=None):
    """Returns out [B,S,Hq,D]; updates the caches in place."""
    lib = lib or load()
    q, k, v = _u16(q), _u16(k), _u16(v)
    out = np.zeros_like(q)
    _check(lib.oracle_prefill(ctypes.byref(cfg_of(shape)), q, k, v, q.shape[1], _u16(k_cache),
                              _u16(v_cache), out), "prefill")
    return out


def prefill_kv(shape, q, k, v, hist_len: int, k_cache, v_cache, lib=None):
    lib = lib or load()
    q, k, v = _u16(q), _u16(k), _u16(v)
    out = np.zeros_like(q)
    _check(lib.oracle_prefill_kv(ctypes.byref(cfg_of(shape)), q, k, v, int(hist_len), q.shape[1],
                                 _u16(k_cache), _u16(v_cache), out), "prefill_kv")
    return out


def decode(shape, q, k, v, hist_len, k_cache, v_cache, lib=None):
    lib = lib or load()
    q, k, v = _u16(q), _u16(k), _u16(v)
    out = np.zeros_like(q)
    h = np.ascontiguousarray(hist_len, dtype=np.int32)
    _check(lib.oracle_decode(ctypes.byref(cfg_of(shape)), q, k, v, h, _u16(k_cache), _u16(v_cache), out),
           "decode")
    return out


def append(shape, k, v, hist, k_cache, v_cache, lib=None):
    """RoPE + in-place cache append of every new token (hist: int or [B])."""
    lib = lib or load()
    k, v = _u16(k), _u16(v)
    h = np.broadcast_to(np.asarray(hist, dtype=np.int32), (shape.batch,)).copy()
    _check(lib.oracle_append(ctypes.byref(cfg_of(shape)), k, v, h, k.shape[1], k.shape[1], _u16(k_cache),
                             _u16(v_cache)), "append")


def attend_rows_parallel(shape, q, hist, k_cache, v_cache, rows, threads=None, lib=None):
    """attend_rows on several host cores: the rows are cut into contiguous blocks and each
    block is one call of the same C routine on its own thread (ctypes releases the GIL,
    and the routine keeps all of its state on its own stack and heap).  Row by row the
    arithmetic is that of attend_rows; only whole rows are distributed."""
    from concurrent.futures import ThreadPoolExecutor
    lib = lib or load()
    r = np.ascontiguousarray(rows, dtype=np.int32).reshape(-1, 3)
    n = max(1, min(int(threads or os.cpu_count() or 1), len(r)))
    out = np.zeros((r.shape[0], shape.head_dim), np.uint16)
    blocks = [ix for ix in np.array_split(np.arange(len(r)), n) if len(ix)]

    def run(ix):
        out[ix] = attend_rows(shape, q, hist, k_cache, v_cache, r[ix], lib=lib)

    with ThreadPoolExecutor(max_workers=n) as ex:
        list(ex.map(run, blocks))
    return out


def attend_rows(shape, q, hist, k_cache, v_cache, rows, lib=None):
    """Output rows for the (b, i, h) triples in ``rows`` over caches that already hold the chunk."""
    lib = lib or load()
    q = _u16(q)
    h = np.broadcast_to(np.asarray(hist, dtype=np.int32), (shape.batch,)).copy()
    r = np.ascontiguousarray(rows, dtype=np.int32).reshape(-1, 3)
    out = np.zeros((r.shape[0], shape.head_dim), np.uint16)
    _check(lib.oracle_attend(ctypes.byref(cfg_of(shape)), q, h, q.shape[1], q.shape[1], _u16(k_cache),
                             _u16(v_cache), out, r.shape[0], r.ctypes.data_as(ctypes.c_void_p)), "attend")
    return out


def prompt(shape, q, k, v, hist_len: int, seg_len: int, k_cache, v_cache, lib=None):
    """Section 4.1, third scenario: a prompt in segments of ``seg_len`` tokens, the
    first by prefill (no history; scenario 1) or prefill_kv (scenario 2), every later
    one by prefill_kv over all positions before it.  q [B,P,Hq,D], k/v [B,P,Hkv,D];
    returns out [B,P,Hq,D] and updates the caches in place."""
    P = q.shape[1]
    outs = []
    for s0 in range(0, P, seg_len):
        sl = slice(s0, min(P, s0 + seg_len))
        qs, ks, vs = (np.ascontiguousarray(a[:, sl]) for a in (q, k, v))
        if hist_len + s0 == 0:
            outs.append(prefill(shape, qs, ks, vs, k_cache, v_cache, lib=lib))
        else:
            outs.append(prefill_kv(shape, qs, ks, vs, hist_len + s0, k_cache, v_cache, lib=lib))
    return np.concatenate(outs, axis=1)


def decode_steps(shape, q, k, v, hist_len, k_cache, v_cache, lib=None):
    """Section 4.5, steps 3-5 restricted to attention: decode steps in a row, step t's
    token of sequence b at position hist_len[b] + t.  q [n,B,1,Hq,D], k/v [n,B,1,Hkv,D];
    returns out [n,B,1,Hq,D] and updates the caches in place."""
    h = np.asarray(hist_len, dtype=np.int64)
    return np.stack([decode(shape, q[t], k[t], v[t], (h + t).astype(np.int32), k_cache, v_cache, lib=lib)
                     for t in range(q.shape[0])])


def decode_multi(shape, q, k, v, hist_len, k_cache, v_cache, lib=None):
    """Decode of n new tokens per sequence (Section 4.4 with n > 1): sequence b's token i
    takes position hist_len[b] + i and attends causally to slots [0, hist_len[b] + i] --
    for each sequence exactly prefill_kv of its n tokens over its own history length.
    q [B,n,Hq,D], k/v [B,n,Hkv,D]; returns out [B,n,Hq,D] and updates the caches in place."""
    import dataclasses
    one = dataclasses.replace(shape, batch=1)
    h = np.asarray(hist_len, dtype=np.int64).reshape(-1)
    out = np.zeros_like(_u16(q))
    for b in range(shape.batch):
        out[b:b + 1] = prefill_kv(one, q[b:b + 1], k[b:b + 1], v[b:b + 1], int(h[b]), k_cache[b:b + 1],
                                  v_cache[b:b + 1], lib=lib)
    return out
