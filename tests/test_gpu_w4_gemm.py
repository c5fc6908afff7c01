"""GPU parity of the W4BF16 weight GEMM of the prefill-side projections (attn_w4bf16_gemm)
against the oracle (oracle/w4_oracle.py: gemm_bf16w, each weight rounded once to bf16; pinned
in tests/w4_oracle_pins.py).

Bound: |y - ref| <= 2^-8 |ref| + 2^-18 A, A = sum_k |x| |W_bf16|: the weights are the same
bf16 values on both sides (the decode rounds exactly as the oracle does), the products are
exact and the sums float on the tensor cores; 2^-8 covers the rounding of y.
Cases: one token, a ragged last token tile, several feature tiles, one input group, and a
sampled check at the size of an 8B-class stacked QKV projection over a 4096-token chunk.
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


def run(torch, codes, scales, zeros, x):
    from paper_2607_15865_gb300.w4 import pack_codes, pack_tiles, w4bf16_gemm
    tiles = torch.from_numpy(pack_tiles(pack_codes(codes), scales, zeros)).cuda()
    xd = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).cuda().view(torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = w4bf16_gemm(tiles, xd, codes.shape[0], err=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return y.view(torch.int16).cpu().numpy().view(np.uint16)


def check(codes, scales, zeros, x, y):
    ref = W.gemm_bf16w(codes, scales, zeros, x)
    a = np.abs(W.bf16_to_f64(x)) @ np.abs(W.bf16_to_f64(W.dequant_bf16(codes, scales, zeros))).T
    got = W.bf16_to_f64(y)
    err = np.abs(got - ref)
    assert np.isfinite(got).all()
    assert (err <= 2.0 ** -8 * np.abs(ref) + 2.0 ** -18 * a).all(), f"max err {err.max():.3e}"


def mat(tag, N, K):
    codes = gen.uint4_codes("w4gemm", f"{tag}_c", (N, K))
    zeros = gen.uint4_codes("w4gemm", f"{tag}_z", (N, K // 128))
    scales = gen.normal_bf16("w4gemm", f"{tag}_s", (N, K // 128), 0.02)
    return codes, scales, zeros


CASES = [("t1", 1, 128, 256), ("t100_ragged", 100, 256, 1024), ("t128", 128, 128, 128),
         ("t300_three_token_tiles", 300, 384, 512), ("t257_k2048", 257, 128, 2048)]


@pytest.mark.parametrize("tag,T,N,K", CASES, ids=[c[0] for c in CASES])
def test_w4_gemm_matches_oracle(torch, tag, T, N, K):
    codes, scales, zeros = mat(tag, N, K)
    x = gen.normal_bf16("w4gemm", f"{tag}_x", (T, K), 1.0)
    check(codes, scales, zeros, x, run(torch, codes, scales, zeros, x))


def test_w4_gemm_full_size_sampled(torch):
    """T = 4096 tokens through an 8B-class stacked QKV projection (N = 6144, K = 4096): the
    oracle on 24 sampled tokens (first, last and random) times every feature."""
    T, N, K = 4096, 6144, 4096
    codes, scales, zeros = mat("big", N, K)
    x = gen.normal_bf16("w4gemm", "big_x", (T, K), 1.0)
    y = run(torch, codes, scales, zeros, x)
    rng = np.random.default_rng(11)
    rows = np.unique(np.concatenate([[0, T - 1], rng.integers(0, T, 22)]))
    check(codes, scales, zeros, x[rows], y[rows])


def test_w4_gemm_rejects_bad_arguments(torch):
    from paper_2607_15865_gb300 import _lib
    lib = _lib.load()
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    p = buf.data_ptr()
    for args in [(None, p, 1, 128, 128, p, None), (p, p, 0, 128, 128, p, None), (p, p, 1, 64, 128, p, None),
                 (p, p, 1, 128, 192, p, None), (p + 8, p, 1, 128, 128, p, None), (p, p + 8, 1, 128, 128, p, None),
                 (p, p, 1, 128, 128, p + 8, None), (p, p, 65535 * 128 + 1, 128, 128, p, None)]:
        assert lib.attn_w4bf16_gemm(*args, None) == _lib.ATTN_EINVAL, args
