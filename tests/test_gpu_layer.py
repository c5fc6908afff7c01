"""GPU parity of the block around attention (Listing 1) for decode with W4BF16 weights:
the fused GEMV parts (RMSNorm of x, residual, split output) and attn_decode_layer
(input_layernorm -> stacked QKV projection -> RoPE + cache append + attention -> o_proj +
residual), against the oracle of oracle/w4_oracle.py (pinned in test_w4_oracle.py).

Bounds.  A GEMV output: 2^-8 |ref| + 2^-18 A as in test_gpu_w4.py, plus, when x is
normalised in the kernel, 2^-5 max_k |xn_k W_nk|: the kernel forms RMSNorm in float and the
oracle in float64, so an element of xn whose value lies within float rounding of a bf16
rounding boundary may land one bf16 step apart (each such element moves y by at most
2^-7 |xn_k W_nk|; the allowance covers four of them).  The layer's output h: 2^-8 |h| plus
2e-2 of the rms of the block's update (h - x) over the row: q, k, v and o are bf16 values
that can differ by a step where the two float paths straddle a rounding boundary, and the
attention stage's own bar is 1e-2 relative.  The appended cache slots: 2^-7 of the slot's
largest magnitude; every other slot bit-exact.
"""
import numpy as np
import pytest

from oracle import w4_oracle as W
from synthetic import gen
from synthetic import workloads as wl
from synthetic.workloads import Shape

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as t
    assert t.cuda.is_available(), "GPU tests need a CUDA device"
    import __graft_entry__
    __graft_entry__.build()
    return t


def dev_bf16(torch, bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def host_bits(t):
    import torch
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def mat(tag, N, K):
    codes = gen.uint4_codes("w4layer", f"{tag}_c", (N, K))
    zeros = gen.uint4_codes("w4layer", f"{tag}_z", (N, K // 128))
    scales = gen.normal_bf16("w4layer", f"{tag}_s", (N, K // 128), 0.02) & np.uint16(0x7FFF)
    return codes, scales, zeros


def tiles_of(torch, m):
    from paper_2607_15865_gb300.w4 import pack_codes, pack_tiles
    codes, scales, zeros = m
    return torch.from_numpy(pack_tiles(pack_codes(codes), scales, zeros)).cuda()


def a_bound(codes, scales, zeros, xb):
    q = np.asarray(codes, np.float64)
    z = np.repeat(np.asarray(zeros, np.float64), W.GROUP, axis=-1)
    s = np.abs(np.repeat(W.bf16_to_f64(scales), W.GROUP, axis=-1))
    return np.abs(W.bf16_to_f64(xb)) @ ((256.0 + q + z) * s).T


def flip_allowance(codes, scales, zeros, xn):
    w = np.abs(W.dequant(codes, scales, zeros))
    return 2.0 ** -5 * np.max(np.abs(W.bf16_to_f64(xn))[:, None, :] * w[None, :, :], axis=-1)


FUSED = [("m1", 1, 200, 1024), ("m3", 3, 96, 4096), ("m8", 8, 64, 2048), ("m11_two_passes", 11, 48, 1024)]


@pytest.mark.parametrize("tag,M,N,K", FUSED, ids=[c[0] for c in FUSED])
def test_fused_gemv_rmsnorm_and_residual(torch, tag, M, N, K):
    from paper_2607_15865_gb300.w4 import w4bf16_gemv_fused
    m = mat(tag, N, K)
    x = gen.normal_bf16("w4layer", f"{tag}_x", (M, K), 1.0)
    gamma = gen.normal_bf16("w4layer", f"{tag}_g", (K,), 0.5)
    res = gen.normal_bf16("w4layer", f"{tag}_r", (M, N), 1.0)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = w4bf16_gemv_fused(tiles_of(torch, m), dev_bf16(torch, x), N, rms_gamma=dev_bf16(torch, gamma), rms_eps=1e-6,
                          residual=dev_bf16(torch, res), err=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    xn = W.rmsnorm(x, gamma, 1e-6)
    ref = W.bf16_to_f64(res) + W.gemv(*m, xn)
    got = W.bf16_to_f64(host_bits(y))
    bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -18 * a_bound(*m, xn) + flip_allowance(*m, xn)
    assert (np.abs(got - ref) <= bound).all(), np.abs(got - ref).max()


def test_fused_gemv_split_matches_unsplit_bits(torch):
    from paper_2607_15865_gb300.w4 import w4bf16_gemv, w4bf16_gemv_fused
    M, N, K = 3, 384, 1024
    m = mat("split", N, K)
    t = tiles_of(torch, m)
    x = dev_bf16(torch, gen.normal_bf16("w4layer", "split_x", (M, K), 1.0))
    whole = w4bf16_gemv(t, x, N)
    q, k, v = w4bf16_gemv_fused(t, x, N, split=(256, 320))
    torch.cuda.synchronize()
    wb = host_bits(whole)
    assert (host_bits(q) == wb[:, :256]).all() and (host_bits(k) == wb[:, 256:320]).all()
    assert (host_bits(v) == wb[:, 320:]).all()


def test_fused_gemv_rejects_bad_parts(torch):
    from paper_2607_15865_gb300 import _lib
    lib = _lib.load()
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    call = lambda g, eps, r, n0, y1, n1, y2: lib.attn_w4bf16_gemv_fused(p, p, 1, 64, 128, g, eps, r, p, n0, y1, n1,
                                                                         y2, None, 0, None)
    assert call(p, 1e-6, p, 16, p, 32, p) == _lib.ATTN_OK
    torch.cuda.synchronize()
    for args in [(p + 4, 1e-6, None, 0, None, 0, None), (p, -1.0, None, 0, None, 0, None),
                 (p, float("nan"), None, 0, None, 0, None), (None, 0.0, p + 1, 0, None, 0, None),
                 (None, 0.0, None, 16, p, 32, None), (None, 0.0, None, 0, p, 32, p), (None, 0.0, None, 32, p, 32, p),
                 (None, 0.0, None, 16, p, 64, p)]:
        assert call(*args) == _lib.ATTN_EINVAL, args


LAYERS = [
    ("b2_g4_d128", Shape("w4l_a", 2, 8, 2, 128, 1024, 1.0e6), 1024, [100, 900]),
    ("b3_g1_d64", Shape("w4l_b", 3, 4, 4, 64, 512, 1.0e4), 512, [0, 17, 300]),
    ("b1_g5_d128_long", Shape("w4l_c", 1, 40, 8, 128, 8192, 1.0e6), 5120, [8000]),
]


def layer_inputs(shape, tag, hidden, hist):
    D = shape.head_dim
    qd, kd = shape.n_q_heads * D, shape.n_kv_heads * D
    x = gen.normal_bf16("w4layer", f"{tag}_x", (shape.batch, hidden), 1.0)
    gamma = gen.normal_bf16("w4layer", f"{tag}_g", (hidden,), 0.5)
    wqkv, wo = mat(f"{tag}_qkv", qd + 2 * kd, hidden), mat(f"{tag}_o", hidden, qd)
    kc, vc = wl.cache(shape, f"{tag}_cache", int(max(hist)), fill="random")
    return x, gamma, wqkv, wo, np.asarray(hist, np.int32), kc, vc


def check_layer(shape, hist, h, kc_gpu, vc_gpu, href, kc_ref, vc_ref, x):
    got, ref = W.bf16_to_f64(h), W.bf16_to_f64(href)
    upd = np.sqrt(np.mean((ref - W.bf16_to_f64(x)) ** 2, axis=-1, keepdims=True))
    assert (np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 2e-2 * upd).all(), np.abs(got - ref).max()
    for gpu, ref_c in ((kc_gpu, kc_ref), (vc_gpu, vc_ref)):
        for b in range(shape.batch):
            s = int(hist[b])
            a, r = W.bf16_to_f64(gpu[b, :, s]), W.bf16_to_f64(ref_c[b, :, s])
            assert (np.abs(a - r) <= 2.0 ** -7 * np.abs(r).max()).all()
            other = np.ones(shape.max_len, bool)
            other[s] = False
            assert (gpu[b][:, other] == ref_c[b][:, other]).all()


@pytest.mark.parametrize("tag,shape,hidden,hist", LAYERS, ids=[c[0] for c in LAYERS])
def test_decode_layer_matches_oracle(torch, tag, shape, hidden, hist):
    from paper_2607_15865_gb300.attention import Attention
    x, gamma, wqkv, wo, hl, kc, vc = layer_inputs(shape, tag, hidden, hist)
    kr, vr = kc.copy(), vc.copy()
    href = W.decode_layer(shape, x, gamma, 1e-6, wqkv, wo, hl, kr, vr)
    attn = Attention.for_shape(shape)
    gk, gv = dev_bf16(torch, kc), dev_bf16(torch, vc)
    xd = dev_bf16(torch, x)
    h = attn.decode_layer(xd, dev_bf16(torch, gamma), 1e-6, tiles_of(torch, wqkv), tiles_of(torch, wo),
                          torch.from_numpy(hl).cuda(), gk, gv, weights_static=True)
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    check_layer(shape, hl, host_bits(h), host_bits(gk).reshape(kc.shape), host_bits(gv).reshape(vc.shape),
                href, kr, vr, x)
    attn.close()


def test_decode_layer_in_place_from_a_cuda_graph(torch):
    """h written over x (the residual stream updated in place), the step captured once and
    replayed: the same result as the oracle."""
    from paper_2607_15865_gb300.attention import Attention
    tag, shape, hidden, hist = LAYERS[0]
    x, gamma, wqkv, wo, hl, kc, vc = layer_inputs(shape, tag + "_graph", hidden, hist)
    kr, vr = kc.copy(), vc.copy()
    href = W.decode_layer(shape, x, gamma, 1e-6, wqkv, wo, hl, kr, vr)
    attn = Attention.for_shape(shape)
    gk, gv = dev_bf16(torch, kc), dev_bf16(torch, vc)
    xd, gd = dev_bf16(torch, x), dev_bf16(torch, gamma)
    tq, to = tiles_of(torch, wqkv), tiles_of(torch, wo)
    hd = torch.from_numpy(hl).cuda()
    attn.decode_layer(xd.clone(), gd, 1e-6, tq, to, hd, gk.clone(), gv.clone())  # warm-up outside the capture
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
        attn.decode_layer(xd, gd, 1e-6, tq, to, hd, gk, gv, out=xd, stream=side)
    torch.cuda.current_stream().wait_stream(side)
    gr.replay()
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    check_layer(shape, hl, host_bits(xd), host_bits(gk).reshape(kc.shape), host_bits(gv).reshape(vc.shape),
                href, kr, vr, x)
    attn.close()
