"""Host-side checks of the W4BF16 binding (no GPU): the wrappers refuse host tensors, wrong
dtypes and sizes before anything reaches the library, and the library reports the rows one
launch stages without a device."""
import numpy as np
import pytest
import torch

from paper_2607_15865_gb300 import _lib
from paper_2607_15865_gb300.w4 import TILE_BYTES, pack_codes, pack_tiles, w4bf16_gemm, w4bf16_gemv, w4bf16_gemv_fused


def test_wrappers_refuse_host_tensors_and_bad_shapes():
    tiles = torch.zeros(2 * 2 * TILE_BYTES, dtype=torch.uint8)
    x = torch.zeros(1, 256, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        w4bf16_gemv(tiles, x, 32)  # host tensors
    with pytest.raises(TypeError):
        w4bf16_gemv_fused(tiles, x, 32, rms_gamma=torch.ones(256, dtype=torch.bfloat16))
    with pytest.raises(TypeError):
        w4bf16_gemm(torch.zeros(8 * 2 * TILE_BYTES, dtype=torch.uint8), x, 128)


def test_pack_tiles_rejects_bad_shapes():
    words = pack_codes(np.zeros((20, 256), np.uint8))
    with pytest.raises(ValueError):
        pack_tiles(words, np.zeros((20, 1), np.uint16), np.zeros((20, 2), np.uint8))
    with pytest.raises(ValueError):
        pack_tiles(pack_codes(np.zeros((20, 200), np.uint8)), np.zeros((20, 1), np.uint16), np.zeros((20, 1), np.uint8))
    with pytest.raises(ValueError):
        pack_codes(np.zeros((2, 12), np.uint8))
    assert pack_tiles(words, np.zeros((20, 2), np.uint16), np.zeros((20, 2), np.uint8)).size == 2 * 2 * TILE_BYTES


def test_rows_per_launch_is_a_host_query():
    lib = _lib.load()
    assert lib.attn_w4bf16_rows_per_launch(4096) == 8
    assert lib.attn_w4bf16_rows_per_launch(100) == 0 and lib.attn_w4bf16_rows_per_launch(-128) == 0
    rows = [lib.attn_w4bf16_rows_per_launch(k) for k in range(128, 1 << 17, 128)]
    assert rows == sorted(rows, reverse=True) and rows[-1] == 0 and set(rows) <= {0, 1, 2, 4, 8}


def test_entry_points_check_arguments_before_the_device():
    """Null pointers, bad sizes and flags come back as ATTN_EINVAL without a device call."""
    lib = _lib.load()
    assert lib.attn_w4bf16_gemv(None, None, 1, 8, 128, None, None, 0, None) == _lib.ATTN_EINVAL
    assert lib.attn_w4bf16_gemv(16, 16, 1, 8, 128, 16, None, 4, None) == _lib.ATTN_EINVAL  # unknown flag
    assert lib.attn_w4bf16_gemv(16, 16, 1, 8, 100, 16, None, 0, None) == _lib.ATTN_EINVAL  # K % 128
    assert lib.attn_decode_layer(None, None, None, 0.0, None, None, 128, None, None, None, None, 0,
                                 None) == _lib.ATTN_EINVAL
    assert lib.attn_w4bf16_gemm(16, 16, 1, 100, 128, 16, None, None) == _lib.ATTN_EINVAL  # N % 128
    assert lib.attn_w4bf16_gemm(16, 16, 0, 128, 128, 16, None, None) == _lib.ATTN_EINVAL  # no tokens


def test_tile_stream_round_trips_for_any_shape():
    """Packer (product), writer and reader (oracle) agree for any row count and group count."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")
    from oracle import w4_oracle as W

    @hyp.settings(max_examples=40, deadline=None)
    @hyp.given(st.integers(1, 70), st.integers(1, 5), st.integers(0, 2 ** 31 - 1))
    def prop(N, ng, seed):
        rng = np.random.default_rng(seed)
        K = 128 * ng
        codes = rng.integers(0, 16, (N, K), dtype=np.uint8)
        scales = rng.integers(0, 1 << 16, (N, ng), dtype=np.uint16)
        zeros = rng.integers(0, 16, (N, ng), dtype=np.uint8)
        buf = pack_tiles(pack_codes(codes), scales, zeros)
        assert buf.size == (N + 15) // 16 * ng * TILE_BYTES
        c, s, z = W.unpack_tiles(buf, N, K)
        assert (c == codes).all() and (s == scales).all() and (z == zeros).all()
        assert (buf == W.write_tiles(codes, scales, zeros)).all()  # byte for byte, padding included

    prop()
