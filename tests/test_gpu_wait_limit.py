"""Failure detection on the GPU without a fault: a bounded wait that runs out.

Every wait inside the library's kernels gives up after a time limit (attn_set_wait_limit;
1 s by default), records ATTN_DEVERR_TIMEOUT, lets the copies and tensor-core work it has
already issued finish, releases its tensor memory and returns.  Here the limit is set to
1 ns, so the kernels of a prefill_kv call and of a decode call give up at their first wait
that is not already satisfied.  The test checks that the calls return, that the device
error word reports the timeout, that the CUDA context is still usable, and that the same
context, with the default limit restored, computes both stages again within the parity
bar of the oracle.  (The outputs of the calls that gave up are undefined.)
"""
import numpy as np
import pytest

from oracle import oracle as O
from synthetic import workloads as w
from synthetic.workloads import Shape
from tests.gpu_util import assert_cache, assert_out_close, to_dev, to_host

pytestmark = pytest.mark.gpu

DEVERR_TIMEOUT = 2

# head_dim 128: flash_fwd with a split tail and the tensor-core decode (its fused merge
# and counters); head_dim 64: flash_fwd and the CUDA-core decode with its merge kernel.
CASES = [
    ("d128", Shape("wl128", 2, 8, 2, 128, 1024, 1.0e4), 300, 333),
    ("d64", Shape("wl64", 1, 4, 2, 64, 640, 1.0e4), 200, 150),
]


@pytest.fixture(scope="module")
def torch():
    import torch as t
    assert t.cuda.is_available(), "GPU tests need a CUDA device"
    import __graft_entry__
    __graft_entry__.build()
    return t


def run_stages(torch, attn, shape, hist, q, k, v, dq, dk, dv, kc, vc):
    """prefill_kv of the chunk over `hist` history tokens, then one decode step at
    hist + chunk for every sequence; returns (chunk out, decode out, k cache, v cache)."""
    gk, gv = to_dev(kc), to_dev(vc)
    out = attn.prefill_kv(to_dev(q), to_dev(k), to_dev(v), hist, gk, gv)
    lens = torch.full((shape.batch,), hist + q.shape[1], dtype=torch.int32, device="cuda")
    dout = attn.decode(to_dev(dq), to_dev(dk), to_dev(dv), lens, gk, gv)
    torch.cuda.synchronize()
    return to_host(out), to_host(dout), to_host(gk), to_host(gv)


@pytest.mark.parametrize("name,shape,hist,chunk", CASES, ids=[c[0] for c in CASES])
def test_wait_limit_runs_out_and_the_context_recovers(torch, name, shape, hist, chunk):
    from paper_2607_15865_gb300.attention import Attention
    q, k, v = w.tokens(shape, "waitlim", chunk + 1)
    q, dq = q[:, :chunk].copy(), q[:, chunk:].copy()
    k, dk = k[:, :chunk].copy(), k[:, chunk:].copy()
    v, dv = v[:, :chunk].copy(), v[:, chunk:].copy()
    kc, vc = w.cache(shape, "waitlim", hist, fill="zero")
    rk, rv = kc.copy(), vc.copy()
    ref = O.prefill_kv(shape, q, k, v, hist, rk, rv)
    ref_dec = O.decode(shape, dq, dk, dv, np.full(shape.batch, hist + chunk, np.int32), rk, rv)

    attn = Attention.for_shape(shape)
    try:
        # 1 ns: the kernels give up at their first wait that is not already satisfied
        attn.set_wait_limit(1)
        run_stages(torch, attn, shape, hist, q, k, v, dq, dk, dv, kc, vc)
        flags = attn.device_error()  # reads and clears the word
        assert flags & DEVERR_TIMEOUT, f"{name}: no wait ran out (error word {flags})"
        # the context is usable: the default limit again, the same calls on fresh caches
        attn.set_wait_limit(0)
        out, dout, gk, gv = run_stages(torch, attn, shape, hist, q, k, v, dq, dk, dv, kc, vc)
        assert attn.device_error() == 0, f"{name}: error word set after the limit was restored"
        assert_out_close(out, ref, f"{name} prefill_kv after recovery")
        assert_out_close(dout, ref_dec, f"{name} decode after recovery")
        assert_cache(gk, gv, rk, rv, kc, vc, [(hist, hist + chunk + 1)] * shape.batch, f"{name} caches")
    finally:
        attn.set_wait_limit(0)
        attn.close()
