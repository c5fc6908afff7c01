"""GPU parity of the block around attention for a prefill / prefill_kv chunk (Listing 1,
Sections 4.2-4.3) with W4BF16 weights: attn_prefill_layer (RMSNorm pre-pass -> stacked QKV
GEMM split three ways -> RoPE + cache append + causal attention -> o_proj GEMM + residual)
against oracle.w4_oracle.prefill_layer (pinned in test_w4_oracle.py).

Bounds.  The block's update u = h - x is linear in the attention output through o_proj, so
it carries the attention stage's own bar: the error norm of u at most 1e-2 of the norm of
u (that bar is set by the bf16 rounding of P and of the output, 2^-9 each; q, k, v also
land one bf16 step apart where the float and float64 paths straddle a rounding boundary).
Over a chunk, o_proj sums hundreds of such bf16-step differences per element, so each
element of h is checked only against 2^-8 |h| + 0.25 rms(u) of its row: a guard against
misplaced rows or columns, which the norm would average away.  The appended cache slots
within 2^-7 of the slot's largest magnitude; every other slot bit-exact.
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
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def mat(tag, N, K):
    codes = gen.uint4_codes("w4pre", f"{tag}_c", (N, K))
    zeros = gen.uint4_codes("w4pre", f"{tag}_z", (N, K // 128))
    scales = gen.normal_bf16("w4pre", f"{tag}_s", (N, K // 128), 0.02) & np.uint16(0x7FFF)
    return codes, scales, zeros


def tiles_of(torch, m):
    from paper_2607_15865_gb300.w4 import pack_codes, pack_tiles
    codes, scales, zeros = m
    return torch.from_numpy(pack_tiles(pack_codes(codes), scales, zeros)).cuda()


CHUNKS = [
    # name, shape, hidden, hist, chunk
    ("b2_g4_d128_pkv", Shape("w4p_a", 2, 8, 2, 128, 1024, 1.0e6), 1024, 77, 150),
    ("b1_g2_d64_prefill", Shape("w4p_b", 1, 4, 2, 64, 512, 1.0e4), 256, 0, 200),
    ("b1_g4_d128_hidden4096", Shape("w4p_c", 1, 32, 8, 128, 2048, 5.0e5), 4096, 1536, 512),
]


def chunk_inputs(shape, tag, hidden, hist, S):
    D = shape.head_dim
    qd, kd = shape.n_q_heads * D, shape.n_kv_heads * D
    x = gen.normal_bf16("w4pre", f"{tag}_x", (shape.batch, S, hidden), 1.0)
    gamma = gen.normal_bf16("w4pre", f"{tag}_g", (hidden,), 0.5)
    wqkv, wo = mat(f"{tag}_qkv", qd + 2 * kd, hidden), mat(f"{tag}_o", hidden, qd)
    kc, vc = wl.cache(shape, f"{tag}_cache", hist, fill="random")
    return x, gamma, wqkv, wo, kc, vc


def check_chunk(shape, hist, S, h, kc_gpu, vc_gpu, href, kc_ref, vc_ref, x):
    got, ref = W.bf16_to_f64(h), W.bf16_to_f64(href)
    u = ref - W.bf16_to_f64(x)
    rel_u = np.linalg.norm(got - ref) / np.linalg.norm(u)
    err = np.abs(got - ref)
    print(f"[parity] prefill block h: max-abs {err.max():.3e}, error norm / update norm {rel_u:.3e}")
    assert rel_u <= 1e-2, rel_u
    rms_u = np.sqrt(np.mean(u ** 2, axis=-1, keepdims=True))
    assert (err <= 2.0 ** -8 * np.abs(ref) + 0.25 * rms_u).all(), err.max()
    for gpu, ref_c in ((kc_gpu, kc_ref), (vc_gpu, vc_ref)):
        for b in range(shape.batch):
            a, r = W.bf16_to_f64(gpu[b, :, hist:hist + S]), W.bf16_to_f64(ref_c[b, :, hist:hist + S])
            assert (np.abs(a - r) <= 2.0 ** -7 * np.abs(r).max(axis=-1, keepdims=True)).all()
            other = np.ones(shape.max_len, bool)
            other[hist:hist + S] = False
            assert (gpu[b][:, other] == ref_c[b][:, other]).all()


@pytest.mark.parametrize("tag,shape,hidden,hist,S", CHUNKS, ids=[c[0] for c in CHUNKS])
def test_prefill_layer_matches_oracle(torch, tag, shape, hidden, hist, S):
    from paper_2607_15865_gb300.attention import Attention
    x, gamma, wqkv, wo, kc, vc = chunk_inputs(shape, tag, hidden, hist, S)
    kr, vr = kc.copy(), vc.copy()
    href = W.prefill_layer(shape, x, gamma, 1e-6, wqkv, wo, hist, kr, vr)
    attn = Attention.for_shape(shape)
    gk, gv = dev_bf16(torch, kc), dev_bf16(torch, vc)
    h = attn.prefill_layer(dev_bf16(torch, x), dev_bf16(torch, gamma), 1e-6, tiles_of(torch, wqkv),
                           tiles_of(torch, wo), hist, gk, gv)
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    check_chunk(shape, hist, S, host_bits(h), host_bits(gk).reshape(kc.shape), host_bits(gv).reshape(vc.shape),
                href, kr, vr, x)
    attn.close()


def test_prefill_layer_in_place_from_a_cuda_graph(torch):
    """h written over x with a caller-owned workspace, the chunk captured once and replayed."""
    from paper_2607_15865_gb300.attention import Attention
    tag, shape, hidden, hist, S = CHUNKS[0]
    x, gamma, wqkv, wo, kc, vc = chunk_inputs(shape, tag + "_graph", hidden, hist, S)
    kr, vr = kc.copy(), vc.copy()
    href = W.prefill_layer(shape, x, gamma, 1e-6, wqkv, wo, hist, kr, vr)
    attn = Attention.for_shape(shape)
    gk, gv = dev_bf16(torch, kc), dev_bf16(torch, vc)
    xd, gd = dev_bf16(torch, x), dev_bf16(torch, gamma)
    tq, to = tiles_of(torch, wqkv), tiles_of(torch, wo)
    ws = torch.empty(attn.prefill_layer_workspace(hidden, S), dtype=torch.uint8, device="cuda")
    attn.prefill_layer(xd.clone(), gd, 1e-6, tq, to, hist, gk.clone(), gv.clone(), workspace=ws)  # warm-up
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
        attn.prefill_layer(xd, gd, 1e-6, tq, to, hist, gk, gv, out=xd, workspace=ws, stream=side)
    torch.cuda.current_stream().wait_stream(side)
    gr.replay()
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    check_chunk(shape, hist, S, host_bits(xd), host_bits(gk).reshape(kc.shape), host_bits(gv).reshape(vc.shape),
                href, kr, vr, x)
    attn.close()


def test_prefill_layer_rejects_bad_arguments(torch):
    from paper_2607_15865_gb300 import _lib
    from paper_2607_15865_gb300.attention import Attention
    shape = CHUNKS[1][1]
    attn = Attention.for_shape(shape)
    lib, ctx = _lib.load(), attn._ctx
    buf = torch.zeros(1 << 22, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    need = lib.attn_prefill_layer_workspace(ctx, 256, 16)
    assert need > 0 and lib.attn_prefill_layer_workspace(ctx, 0, 16) == 0
    call = lambda hidden, hist, S, ws, nbytes, eps=1e-6: lib.attn_prefill_layer(
        ctx, p, p, eps, p, p, hidden, hist, S, p, p, p, ws, nbytes, None)
    for args in [(200, 0, 16, p, need), (256, 0, 0, p, need), (256, 500, 16, p, need), (256, -1, 16, p, need),
                 (256, 0, 16, p + 16, need), (256, 0, 16, p, need - 1), (256, 0, 16, None, need),
                 (256, 0, 16, p, need, -1.0), (256, 0, 16, p, need, float("inf"))]:
        assert call(*args) == _lib.ATTN_EINVAL, args
    attn.close()
