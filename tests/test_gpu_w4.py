"""GPU parity of the W4BF16 weight-only GEMV (attn_w4bf16_gemv), the decode-side
weight stream of the paper's W4BF16 deployment (Section 5.1, Section 5.2).

Compared with the float64 oracle (oracle/w4_oracle.py, pinned in test_w4_oracle.py).
The kernel's arithmetic: per 128-input group and row, D = sum (128 + q) x with exact
products and f32 sums (tensor-core accumulation), minus (128 + z) * (f32 sum of x over
the group), times s, summed in f32 over the groups; y rounded to bf16.  Bound used:
  |y - ref| <= 2^-8 |ref| + 2^-18 A,  A = sum_k |x| ((128 + q) + (128 + z)) s:
2^-8 covers the bf16 rounding of y (half an ulp is 2^-9 relative); A bounds every
partial sum the kernel forms, and 2^-18 A is several times the f32 rounding seen in
sums of that size (the worst case, (K/128 + 133) 2^-24 A, would hide real errors).

Cases: one to sixteen activation rows (the kernel is built for 1, 2, 4 and 8 rows, more
take further passes), rows of weights that do not fill a unit of 16, K that splits
unevenly across the warps of a CTA and into stages, the largest K one launch stages, a
sampled check at a weight size beyond the L2 cache, and the argument checks.
"""
import numpy as np
import pytest

from oracle import w4_oracle as W
from synthetic import gen

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as t
    assert t.cuda.is_available(), "GPU tests need a CUDA device"
    import __graft_entry__
    __graft_entry__.build()
    return t


def make(tag, M, N, K):
    codes = gen.uint4_codes("w4gpu", f"{tag}_codes", (N, K))
    zeros = gen.uint4_codes("w4gpu", f"{tag}_zeros", (N, K // 128))
    scales = gen.normal_bf16("w4gpu", f"{tag}_scales", (N, K // 128), 0.02) & np.uint16(0x7FFF)
    x = gen.normal_bf16("w4gpu", f"{tag}_x", (M, K), 1.0)
    return codes, zeros, scales, x


def run(torch, words, zeros, scales, x):
    """The kernel on row words [N, K/8] (packed into the tile stream here)."""
    from paper_2607_15865_gb300.w4 import pack_tiles, w4bf16_gemv
    tiles = torch.from_numpy(pack_tiles(words, scales, zeros)).cuda()
    xd = torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = w4bf16_gemv(tiles, xd, words.shape[0], err=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return y.view(torch.int16).cpu().numpy().view(np.uint16)


def partial_sum_bound(codes, scales, zeros, x):
    """A[m, n] = sum_k |x[m, k]| ((128 + q[n, k]) + (128 + z[n, k // 128])) s[n, k // 128]."""
    q = np.asarray(codes, np.float64)
    z = np.repeat(np.asarray(zeros, np.float64), W.GROUP, axis=-1)
    s = np.abs(np.repeat(W.bf16_to_f64(scales), W.GROUP, axis=-1))
    return np.abs(W.bf16_to_f64(x)) @ ((256.0 + q + z) * s).T


def check(codes, zeros, scales, x, y_bits, rows=None):
    codes = codes if rows is None else codes[rows]
    sc = scales if rows is None else scales[rows]
    zp = zeros if rows is None else zeros[rows]
    ref = W.gemv(codes, sc, zp, x)
    got = W.bf16_to_f64(y_bits if rows is None else y_bits[:, rows])
    bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -18 * partial_sum_bound(codes, sc, zp, x)
    err = np.abs(got - ref)
    assert np.isfinite(got).all()
    assert (err <= bound).all(), f"max err {err.max():.3e}, worst ratio {(err / np.maximum(bound, 1e-30)).max():.2f}"


CASES = [
    ("m1_small", 1, 64, 1024),
    ("m1_ragged_rows_and_steps", 1, 131, 4096 + 384),
    ("m1_one_group", 1, 5, 128),
    ("m1_single_row", 1, 1, 128),
    ("m2_fifteen_rows_of_a_tile", 2, 15, 384),
    ("m7_seventeen_rows", 7, 17, 640),
    ("m2", 2, 100, 2048),
    ("m3_in_the_4_row_kernel", 3, 77, 1152),
    ("m4", 4, 256, 4096),
    ("m5_in_the_8_row_kernel", 5, 33, 512),
    ("m8", 8, 300, 3072),
    ("m9_two_passes", 9, 40, 1024),
    ("m16_two_passes", 16, 64, 2048),
    ("m6_k12800_several_passes", 6, 9, 12800),
    ("m8_k16384_several_passes", 8, 20, 16384),
    ("m1_many_units_per_warp", 1, 12000, 256),
    ("m8_many_units_per_warp", 8, 6000, 256),
]


@pytest.mark.parametrize("tag,M,N,K", CASES, ids=[c[0] for c in CASES])
def test_w4_gemv_matches_oracle(torch, tag, M, N, K):
    from paper_2607_15865_gb300.w4 import pack_codes
    codes, zeros, scales, x = make(tag, M, N, K)
    y = run(torch, pack_codes(codes), zeros, scales, x)
    assert y.shape == (M, N)
    check(codes, zeros, scales, x, y)


def k_max():
    """The largest K one launch stages for a single row of x."""
    from paper_2607_15865_gb300 import _lib
    lib = _lib.load()
    k = 128
    while lib.attn_w4bf16_rows_per_launch(k + 128) >= 1:
        k += 128
    return k


def test_w4_gemv_rows_per_launch(torch):
    from paper_2607_15865_gb300 import _lib
    lib = _lib.load()
    assert lib.attn_w4bf16_rows_per_launch(0) == 0 and lib.attn_w4bf16_rows_per_launch(200) == 0
    assert lib.attn_w4bf16_rows_per_launch(4096) == 8
    km = k_max()
    assert km >= 32768 and lib.attn_w4bf16_rows_per_launch(km + 128) == 0
    rows = [lib.attn_w4bf16_rows_per_launch(k) for k in range(128, km + 1, 128)]
    assert all(r in (1, 2, 4, 8) for r in rows) and rows == sorted(rows, reverse=True)


def test_w4_gemv_largest_k(torch):
    from paper_2607_15865_gb300.w4 import pack_codes
    M, N, K = 1, 17, k_max()
    codes, zeros, scales, x = make("kmax", M, N, K)
    check(codes, zeros, scales, x, run(torch, pack_codes(codes), zeros, scales, x))


def test_w4_gemv_beyond_l2_sampled(torch):
    """A 160 MiB code matrix (N = 40960, K = 8192), larger than the L2 cache: rows
    sampled across the matrix, the first and last rows included, against the oracle."""
    M, N, K = 1, 40960, 8192
    words = gen.uint32_words("w4gpu", "big_words", (N, K // 8))
    zeros = gen.uint4_codes("w4gpu", "big_zeros", (N, K // 128))
    scales = gen.normal_bf16("w4gpu", "big_scales", (N, K // 128), 0.02) & np.uint16(0x7FFF)
    x = gen.normal_bf16("w4gpu", "big_x", (M, K), 1.0)
    y = run(torch, words, zeros, scales, x)
    rng = np.random.default_rng(7)
    rows = np.unique(np.concatenate([[0, 1, N - 1], rng.integers(0, N, 61)]))
    check(W.unpack_row_words(words[rows]), zeros[rows], scales[rows], x, y[:, rows])


def test_w4_gemv_zero_points_cancel(torch):
    """codes equal to the zero points give y = 0 up to the f32 rounding of
    (128 + q) x - (128 + z) x, whatever x and s."""
    from paper_2607_15865_gb300.w4 import pack_codes
    M, N, K = 2, 40, 1024
    _, zeros, scales, x = make("zc", M, N, K)
    codes = np.repeat(zeros, 128, axis=1)
    y = run(torch, pack_codes(codes), zeros, scales, x)
    assert (np.abs(W.bf16_to_f64(y)) <= 2.0 ** -18 * partial_sum_bound(codes, scales, zeros, x)).all()


def test_w4_gemv_rejects_bad_arguments(torch):
    from paper_2607_15865_gb300 import _lib
    lib = _lib.load()
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    ok = lib.attn_w4bf16_gemv(p, p, 1, 8, 128, p + 65536, p + 131072, 0, None)
    assert ok == _lib.ATTN_OK
    for args in [(None, p, 1, 8, 128, p, None, 0), (p, None, 1, 8, 128, p, None, 0), (p, p, 1, 8, 128, None, None, 0),
                 (p, p, 0, 8, 128, p, None, 0), (p, p, 1, 0, 128, p, None, 0), (p, p, 1, 8, 64, p, None, 0),
                 (p, p, 1, 8, 200, p, None, 0), (p, p, 1, 8, k_max() + 128, p, None, 0),
                 (p + 8, p, 1, 8, 128, p, None, 0), (p, p + 8, 1, 8, 128, p, None, 0),
                 (p, p, 1, 8, 128, p + 1, None, 0), (p, p, 1, 8, 128, p, p + 2, 0), (p, p, 1, 8, 128, p, None, 2)]:
        assert lib.attn_w4bf16_gemv(*args, None) == _lib.ATTN_EINVAL, args
    torch.cuda.synchronize()
    assert int(buf[131072:131076].view(torch.int32).item()) == 0


@pytest.mark.parametrize("weights_static", [False, True])
def test_w4_gemv_chain_feeds_each_output_forward(torch, weights_static):
    """A chain of GEMVs where each call's x is the previous call's y (dependent launches,
    in a CUDA graph and eagerly): every output against the oracle applied to the input the
    GPU actually fed it.  With weights_static the next matrix is streamed before the
    previous call finishes; x and y must still follow the stream order."""
    from paper_2607_15865_gb300.w4 import pack_codes, pack_tiles, w4bf16_gemv
    M, dims = 2, [1024, 3072, 512, 2048, 1024]
    layers = []
    for i in range(len(dims) - 1):
        K, N = dims[i], dims[i + 1]
        codes, zeros, scales, _ = make(f"chain{i}", 1, N, K)
        tiles = torch.from_numpy(pack_tiles(pack_codes(codes), scales, zeros)).cuda()
        layers.append((codes, zeros, scales, tiles, N))
    x0 = make("chain_x", M, 8, dims[0])[3]
    xs = [torch.from_numpy(x0.view(np.int16)).cuda().view(torch.bfloat16)]
    xs += [torch.empty((M, n), dtype=torch.bfloat16, device="cuda") for n in dims[1:]]
    err = torch.zeros(1, dtype=torch.int32, device="cuda")

    def chain(stream):
        for i, (_, _, _, tiles, N) in enumerate(layers):
            w4bf16_gemv(tiles, xs[i], N, out=xs[i + 1], stream=stream, err=err, weights_static=weights_static)

    def check_all():
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        for i, (codes, zeros, scales, _, _) in enumerate(layers):
            xin = xs[i].view(torch.int16).cpu().numpy().view(np.uint16)
            yout = xs[i + 1].view(torch.int16).cpu().numpy().view(np.uint16)
            check(codes, zeros, scales, xin, yout)

    chain(None)
    check_all()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
        chain(side)
    torch.cuda.current_stream().wait_stream(side)
    for t in xs[1:]:
        t.fill_(float("nan"))
    gr.replay()
    check_all()
