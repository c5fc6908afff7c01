"""The stage calls inside a CUDA graph: captured once, replayed with new inputs.

include/attn.h promises that no stage call allocates, frees or synchronises, so a
serving loop can capture a step (prefill_kv of a chunk, then a decode) into a CUDA
graph and replay it.  The graph is captured once on static device buffers and
replayed twice with new q/k/v and new per-sequence decode lengths written into those
buffers; every replay must match the oracle run on the same inputs in the same order.
"""
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


@pytest.mark.parametrize("shape", [Shape("graph_d128", 2, 8, 2, 128, 512, 1.0e4),
                                   Shape("graph_d64", 2, 6, 3, 64, 384, 1.0e4)], ids=["d128", "d64"])
def test_step_captured_in_a_cuda_graph(torch, shape):
    from paper_2607_15865_gb300.attention import Attention
    hist0, chunk = 100, 64
    attn = Attention.for_shape(shape)
    kc, vc = w.cache(shape, shape.name, hist0, fill="random")
    gk, gv = to_dev(kc), to_dev(vc)
    rk, rv = kc.copy(), vc.copy()

    def inputs(tag, dec_hist):
        qp, kp, vp = w.tokens(shape, f"{tag}_chunk", chunk)
        qd, kd, vd = w.tokens(shape, f"{tag}_dec", 1)
        return (qp, kp, vp), (qd, kd, vd), np.asarray(dec_hist, np.int32)

    # static device buffers, filled before capture with the first replay's inputs
    (qp, kp, vp), (qd, kd, vd), h = inputs("g0", [hist0 + chunk, hist0 + chunk + 5])
    d_qp, d_kp, d_vp = to_dev(qp), to_dev(kp), to_dev(vp)
    d_qd, d_kd, d_vd = to_dev(qd), to_dev(kd), to_dev(vd)
    d_h = torch.from_numpy(h).cuda()
    out_p, out_d = torch.empty_like(d_qp), torch.empty_like(d_qd)

    # warm the context on a scratch copy of the caches (tensor maps, first-launch set-up)
    wk, wv = gk.clone(), gv.clone()
    attn.prefill_kv(d_qp, d_kp, d_vp, hist0, wk, wv, out=out_p)
    attn.decode(d_qd, d_kd, d_vd, d_h, wk, wv, out=out_d)
    torch.cuda.synchronize()
    del wk, wv

    graph = torch.cuda.CUDAGraph()
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            attn.prefill_kv(d_qp, d_kp, d_vp, hist0, gk, gv, out=out_p)
            attn.decode(d_qd, d_kd, d_vd, d_h, gk, gv, out=out_d)
    torch.cuda.current_stream().wait_stream(stream)
    torch.cuda.synchronize()
    # capture records the kernels without running them: the caches are still the initial ones
    assert (to_host(gk) == kc).all() and (to_host(gv) == vc).all()

    written = [set() for _ in range(shape.batch)]
    for rep, (tag, dec_hist) in enumerate([("g0", [hist0 + chunk, hist0 + chunk + 5]),
                                           ("g1", [hist0 + chunk + 9, hist0 + chunk])]):
        (qp, kp, vp), (qd, kd, vd), h = inputs(tag, dec_hist)
        for dst, src in ((d_qp, qp), (d_kp, kp), (d_vp, vp), (d_qd, qd), (d_kd, kd), (d_vd, vd)):
            dst.copy_(torch.from_numpy(src.view(np.int16)))
        d_h.copy_(torch.from_numpy(h))
        graph.replay()
        torch.cuda.synchronize()
        ref_p = O.prefill_kv(shape, qp, kp, vp, hist0, rk, rv)  # appends to rk, rv in place
        ref_d = O.decode(shape, qd, kd, vd, h, rk, rv)
        assert_out_close(to_host(out_p), ref_p, f"{shape.name} graph replay {rep}: prefill_kv")
        assert_out_close(to_host(out_d), ref_d, f"{shape.name} graph replay {rep}: decode")
        for b in range(shape.batch):
            written[b].update(range(hist0, hist0 + chunk))
            written[b].add(int(h[b]))
    assert attn.device_error() == 0
    lo = [min(s_) for s_ in written]
    hi = [max(s_) + 1 for s_ in written]
    assert_cache(to_host(gk), to_host(gv), rk, rv, kc, vc, list(zip(lo, hi)), f"{shape.name} graph cache")
    attn.close()
