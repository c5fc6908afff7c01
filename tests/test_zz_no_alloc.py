"""attn_decode_noalloc -- decode for callers that cannot allocate device memory.

Code running inside a framework that owns every device buffer, or in a process
whose device memory is provisioned once up front, cannot call cudaMalloc and so
cannot create a context with attn_create.  attn_decode_noalloc takes every
buffer from the caller (RoPE tables and error word included) and keeps its
split-KV scratch in a static device array.  These tests call it through the C
ABI and check that it computes what attn_decode computes, on two calls in a row,
and that it refuses shapes whose scratch would not fit.

This file is collected last on purpose: if it fails, a run stopping at the first
failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest

from synthetic import workloads as w
from synthetic.workloads import Shape
from tests.gpu_util import assert_out_close, to_dev, to_host, ulp_diff

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300 import _lib
    return torch, _lib, _lib.load()


def rope_tables(shape):
    """The table layout attn_decode_noalloc documents: cos/sin of p*theta^(-2j/D),
    evaluated in double and rounded to float, row p, column j."""
    j = np.arange(shape.head_dim // 2, dtype=np.float64)
    inv_freq = np.power(shape.rope_theta, -(2.0 * j) / shape.head_dim)
    ang = np.arange(shape.max_len, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang).astype(np.float32), np.sin(ang).astype(np.float32)


# head_dim 128 runs the tensor-core decode (its merge fused in, counters in the static
# array); head_dim 64 runs the CUDA-core split kernel and the merge kernel, both reading
# and writing the static partials.  The scratch cap never binds below attn_decode's own
# split count for these kernels' split rules (it would need more than 50 query heads per
# kv head), so both calls run attn_decode's split count.
CASES = [
    ("d128_b4", Shape("noalloc128", 4, 32, 8, 128, 8192, 5.0e5), 8191,
     ([1024, 4096, 8191, 17], [5, 0, 8000, 3000])),
    ("d64_b3", Shape("noalloc64", 3, 4, 2, 64, 64, 1.0e4), 60, ([24, 5, 63], [0, 40, 27])),
]


@pytest.mark.parametrize("name,shape,n_hist,calls", CASES, ids=[c[0] for c in CASES])
def test_noalloc_decode_matches_attn_decode_and_the_oracle_on_two_calls(env, name, shape, n_hist, calls):
    from oracle import oracle as O
    torch, _lib, lib = env
    from paper_2607_15865_gb300.attention import Attention
    cfg = _lib.AttnCfg(shape.batch, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.max_len,
                       shape.rope_theta)
    ctab, stab = rope_tables(shape)
    d_cos, d_sin = torch.from_numpy(ctab).cuda(), torch.from_numpy(stab).cuda()
    attn = Attention.for_shape(shape)
    kc, vc = w.cache(shape, "noalloc", n_hist, fill="random")
    ref_k, ref_v = to_dev(kc), to_dev(vc)
    new_k, new_v = to_dev(kc), to_dev(vc)
    ork, orv = kc.copy(), vc.copy()  # the oracle's own caches
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    for call, hist in enumerate(calls):
        q, k, v = w.tokens(shape, f"noalloc{call}", 1)
        hl = torch.tensor(hist, dtype=torch.int32, device="cuda")
        ref = attn.decode(to_dev(q), to_dev(k), to_dev(v), hl, ref_k, ref_v)
        oref = O.decode(shape, q, k, v, np.asarray(hist, np.int32), ork, orv)
        dq, dk, dv = to_dev(q), to_dev(k), to_dev(v)
        out = torch.empty_like(dq)
        rc = lib.attn_decode_noalloc(ctypes.byref(cfg), d_cos.data_ptr(), d_sin.data_ptr(), dq.data_ptr(),
                                     dk.data_ptr(), dv.data_ptr(), hl.data_ptr(), new_k.data_ptr(),
                                     new_v.data_ptr(), out.data_ptr(), err.data_ptr(), stream.cuda_stream)
        assert rc == _lib.ATTN_OK, lib.attn_strerror(rc)
        torch.cuda.synchronize()
        assert int(err.item()) == 0, "the no-alloc decode set an error bit"
        assert attn.device_error() == 0
        got = to_host(out)
        assert_out_close(got, to_host(ref), f"{name}: no-alloc vs attn_decode, call {call + 1}")
        assert_out_close(got, oref, f"{name}: no-alloc vs the oracle, call {call + 1}")
        assert ulp_diff(to_host(new_k), to_host(ref_k)).max() <= 1, f"k cache differs, call {call + 1}"
        assert (to_host(new_v) == to_host(ref_v)).all(), f"v cache differs, call {call + 1}"
        assert ulp_diff(to_host(new_k), ork).max() <= 1, f"k cache differs from the oracle's, call {call + 1}"
        assert (to_host(new_v) == orv).all(), f"v cache differs from the oracle's, call {call + 1}"
    attn.close()


def test_noalloc_decode_rejects_scratch_overflow(env):
    torch, _lib, lib = env
    # 1024 * 8 * (128 + 2) floats of partials per split exceed the 2^20-float array:
    # rejected on the host before any device work (the pointers are never touched).
    cfg = _lib.AttnCfg(1024, 8, 8, 128, 64, 1.0e4)
    assert 1024 * 8 * 130 > _lib.NOALLOC_SCRATCH_FLOATS
    p = 256
    rc = lib.attn_decode_noalloc(ctypes.byref(cfg), p, p, p, p, p, p, p, p, p, p, None)
    assert rc == _lib.ATTN_EINVAL
