"""GPU parity of the stage driver (attn_prompt, attn_decode_steps; Sections 4.1 and 4.5).

A long prompt runs in segments (1 prefill + N prefill_kv, or N prefill_kv after a
history) and decode runs several steps per call; every output and the final caches
must match the oracle of the same composition.  The oracle's composition is itself
pinned (tests/test_oracle_driver.py) to one prefill_kv of the whole prompt.  A
conversation of two sessions, the decode loop replayed from a CUDA graph, and the
argument checks follow.
"""
import ctypes

import numpy as np
import pytest

from oracle import oracle as O
from synthetic import workloads as w
from synthetic.workloads import Shape
from tests.gpu_util import assert_cache, assert_out_close, to_dev, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as t
    assert t.cuda.is_available(), "GPU tests need a CUDA device"
    import __graft_entry__
    __graft_entry__.build()
    return t


def step_major(a):
    """[B, n, H, D] token-major -> [n, B, 1, H, D] step-major (contiguous)."""
    return np.ascontiguousarray(a.transpose(1, 0, 2, 3)[:, :, None])


PROMPTS = [
    ("d128_b2_from_empty", Shape("drv1", 2, 8, 2, 128, 1024, 1.0e4), 0, 700, 256),
    ("d128_b1_after_history", Shape("drv2", 1, 10, 2, 128, 2048, 1.0e6), 301, 900, 384),
    ("d64_b2_short_segments", Shape("drv3", 2, 4, 2, 64, 600, 1.0e4), 17, 333, 100),
    ("one_segment", Shape("drv4", 1, 4, 1, 128, 512, 1.0e4), 0, 200, 512),
    ("segments_of_one_token", Shape("drv5", 1, 4, 2, 128, 64, 1.0e4), 5, 9, 1),
]


@pytest.mark.parametrize("name,shape,hist,P,seg", PROMPTS, ids=[p[0] for p in PROMPTS])
def test_prompt_in_segments_matches_oracle(torch, name, shape, hist, P, seg):
    from paper_2607_15865_gb300.attention import Attention
    attn = Attention.for_shape(shape)
    q, k, v = w.tokens(shape, "drv_prompt", P)
    kc, vc = w.cache(shape, "drv_prompt", hist, fill="nan")
    rk, rv = kc.copy(), vc.copy()
    gk, gv = to_dev(kc), to_dev(vc)
    out = attn.prompt(to_dev(q), to_dev(k), to_dev(v), hist, seg, gk, gv)
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    ref = O.prompt(shape, q, k, v, hist, seg, rk, rv)
    assert_out_close(to_host(out), ref, f"{name} out")
    assert_cache(to_host(gk), to_host(gv), rk, rv, kc, vc, [(hist, hist + P)] * shape.batch, f"{name} cache")
    attn.close()


def test_two_session_conversation(torch):
    """Section 4.1 scenario 2: session 1 = prompt + decode loop; session 2 continues
    over everything so far (prompt via prefill_kv) + decode loop; both sequences of
    the batch start at the same length, so the lengths array is shared."""
    from paper_2607_15865_gb300.attention import Attention
    shape = Shape("conv", 2, 8, 2, 128, 1536, 1.0e6)
    attn = Attention.for_shape(shape)
    kc, vc = w.cache(shape, "conv", 0, fill="nan")
    rk, rv = kc.copy(), vc.copy()
    gk, gv = to_dev(kc), to_dev(vc)
    hist = 0
    for sess, (P, seg, n_dec) in enumerate([(530, 256, 6), (410, 128, 5)]):
        q, k, v = w.tokens(shape, f"conv{sess}_prompt", P)
        out = attn.prompt(to_dev(q), to_dev(k), to_dev(v), hist, seg, gk, gv)
        ref = O.prompt(shape, q, k, v, hist, seg, rk, rv)
        torch.cuda.synchronize()
        assert_out_close(to_host(out), ref, f"session {sess} prompt")
        hist += P
        qd, kd, vd = (step_major(a) for a in w.tokens(shape, f"conv{sess}_dec", n_dec))
        hl = np.full(shape.batch, hist, np.int32)
        outd = attn.decode_steps(to_dev(qd), to_dev(kd), to_dev(vd), torch.from_numpy(hl).cuda(), gk, gv)
        refd = O.decode_steps(shape, qd, kd, vd, hl, rk, rv)
        torch.cuda.synchronize()
        assert_out_close(to_host(outd), refd, f"session {sess} decode steps")
        hist += n_dec
    assert attn.device_error() == 0
    assert_cache(to_host(gk), to_host(gv), rk, rv, kc, vc, [(0, hist)] * shape.batch, "conversation cache")
    attn.close()


@pytest.mark.parametrize("shape", [Shape("dsteps_d128", 3, 8, 2, 128, 700, 1.0e4),
                                   Shape("dsteps_d64", 2, 6, 3, 64, 300, 1.0e4)], ids=["d128", "d64"])
def test_decode_steps_mixed_lengths(torch, shape):
    from paper_2607_15865_gb300.attention import Attention
    attn = Attention.for_shape(shape)
    n = 7
    hl = np.array([5, 290, 131][:shape.batch], np.int32)
    kc, vc = w.cache(shape, "dsteps", int(hl.max()), fill="random")
    rk, rv = kc.copy(), vc.copy()
    gk, gv = to_dev(kc), to_dev(vc)
    qd, kd, vd = (step_major(a) for a in w.tokens(shape, "dsteps", n))
    out = attn.decode_steps(to_dev(qd), to_dev(kd), to_dev(vd), torch.from_numpy(hl).cuda(), gk, gv)
    ref = O.decode_steps(shape, qd, kd, vd, hl, rk, rv)
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    assert_out_close(to_host(out), ref, f"{shape.name} decode steps")
    assert_cache(to_host(gk), to_host(gv), rk, rv, kc, vc, [(int(h), int(h) + n) for h in hl], f"{shape.name} cache")
    attn.close()


def test_decode_steps_past_max_len_flag_and_skip(torch):
    """Steps whose position reaches max_len are skipped for that sequence and flagged;
    the steps before them are computed as usual."""
    from paper_2607_15865_gb300 import _lib
    from paper_2607_15865_gb300.attention import Attention
    shape = Shape("dsteps_edge", 2, 4, 2, 128, 256, 1.0e4)
    attn = Attention.for_shape(shape)
    n = 4
    hl = np.array([254, 100], np.int32)  # sequence 0: positions 254, 255, then 256 and 257 are out of range
    kc, vc = w.cache(shape, "dsteps_edge", 254, fill="random")
    rk, rv = kc.copy(), vc.copy()
    gk, gv = to_dev(kc), to_dev(vc)
    qd, kd, vd = (step_major(a) for a in w.tokens(shape, "dsteps_edge", n))
    out = torch.full((n, 2, 1, 4, 128), 0x7F00, dtype=torch.int16, device="cuda")  # sentinel bits
    attn.decode_steps(to_dev(qd), to_dev(kd), to_dev(vd), torch.from_numpy(hl).cuda(), gk, gv, out=out)
    flags = attn.device_error()
    assert flags & _lib.DEVERR_HIST_RANGE
    got = to_host(out)
    rk1, rv1 = None, None
    for t in range(n):
        if t == 2:  # from here on only sequence 1 advances: continue its own oracle cache
            rk1, rv1 = np.ascontiguousarray(rk[1:]), np.ascontiguousarray(rv[1:])
        if t < 2:  # both sequences in range
            ref = O.decode(shape, qd[t], kd[t], vd[t], hl + t, rk, rv)
            assert_out_close(got[t], ref, f"step {t}")
        else:  # sequence 0 out of range: skipped; sequence 1 computed
            assert (got[t][0] == 0x7F00).all(), f"step {t}: out-of-range sequence 0 was written"
            one = Shape("dsteps_edge1", 1, 4, 2, 128, 256, 1.0e4)
            ref1 = O.decode(one, qd[t][1:], kd[t][1:], vd[t][1:], hl[1:] + t, rk1, rv1)
            assert_out_close(got[t][1:], ref1, f"step {t} sequence 1")
    attn.close()


def test_decode_steps_replayed_from_a_cuda_graph(torch):
    from paper_2607_15865_gb300.attention import Attention
    shape = Shape("dsteps_graph", 2, 8, 2, 128, 512, 1.0e4)
    attn = Attention.for_shape(shape)
    n, hist0 = 5, 200
    kc, vc = w.cache(shape, "dgraph", hist0, fill="random")
    gk, gv = to_dev(kc), to_dev(vc)
    rk, rv = kc.copy(), vc.copy()
    qd, kd, vd = (step_major(a) for a in w.tokens(shape, "dgraph0", n))
    d_q, d_k, d_v = to_dev(qd), to_dev(kd), to_dev(vd)
    d_h = torch.from_numpy(np.full(2, hist0, np.int32)).cuda()
    out = torch.empty_like(d_q)
    wk, wv = gk.clone(), gv.clone()
    attn.decode_steps(d_q, d_k, d_v, d_h, wk, wv, out=out)  # warm-up on scratch caches
    torch.cuda.synchronize()
    del wk, wv
    graph = torch.cuda.CUDAGraph()
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            attn.decode_steps(d_q, d_k, d_v, d_h, gk, gv, out=out)
    torch.cuda.current_stream().wait_stream(stream)
    torch.cuda.synchronize()
    hist = hist0
    for rep in range(2):
        qd, kd, vd = (step_major(a) for a in w.tokens(shape, f"dgraph{rep}", n))
        for dst, src in ((d_q, qd), (d_k, kd), (d_v, vd)):
            dst.copy_(torch.from_numpy(src.view(np.int16)))
        hl = np.full(2, hist, np.int32)
        d_h.copy_(torch.from_numpy(hl))
        graph.replay()
        torch.cuda.synchronize()
        ref = O.decode_steps(shape, qd, kd, vd, hl, rk, rv)
        assert_out_close(to_host(out), ref, f"graph replay {rep}")
        hist += n
    assert attn.device_error() == 0
    assert_cache(to_host(gk), to_host(gv), rk, rv, kc, vc, [(hist0, hist)] * 2, "graph cache")
    attn.close()


def test_driver_rejects_bad_arguments(torch):
    from paper_2607_15865_gb300 import _lib
    from paper_2607_15865_gb300.attention import Attention
    shape = Shape("drv_bad", 1, 4, 2, 128, 128, 1.0e4)
    attn = Attention.for_shape(shape)
    q, k, v = (to_dev(a) for a in w.tokens(shape, "bad", 64))
    kc, vc = (to_dev(a) for a in w.cache(shape, "bad", 0))
    with pytest.raises(_lib.AttnError) as e:
        attn.prompt(q, k, v, 65, 32, kc, vc)  # 65 + 64 > max_len
    assert e.value.code == _lib.ATTN_EINVAL
    with pytest.raises(_lib.AttnError) as e:
        attn.prompt(q, k, v, 0, 0, kc, vc)  # empty segments
    assert e.value.code == _lib.ATTN_EINVAL
    lib = attn.lib
    d_h = torch.zeros(1, dtype=torch.int32, device="cuda")
    qd = torch.zeros((1, 1, 1, 4, 128), dtype=torch.int16, device="cuda")
    kd = torch.zeros((1, 1, 1, 2, 128), dtype=torch.int16, device="cuda")
    rc = lib.attn_decode_steps(attn.handle, qd.data_ptr(), kd.data_ptr(), kd.data_ptr(), d_h.data_ptr(), 0,
                               kc.data_ptr(), vc.data_ptr(), qd.data_ptr(), None)
    assert rc == _lib.ATTN_EINVAL
    rc = lib.attn_prompt(attn.handle, q.data_ptr(), k.data_ptr(), v.data_ptr(), 0, 64, 16, kc.data_ptr(),
                         vc.data_ptr(), None, None)
    assert rc == _lib.ATTN_EINVAL
    torch.cuda.synchronize()
    assert (to_host(kc) == 0).all(), "a rejected call wrote the cache"
    attn.close()
