"""Pins of the W4BF16 GEMV oracle (the decode-side weight stream of the paper's W4BF16
deployment, Section 5.1) against what the definition fixes by itself.

  * format: the product's packer and the oracle's reader agree on every code, scale and
    zero point of a matrix whose rows do not fill the last tile, and single values land
    at the byte and bit the documented format names;
  * brute force: y[m, n] = sum_k x[m, k] (q[n, k] - z[n, k // 128]) s[n, k // 128] written
    as plain Python loops on a tiny case;
  * closed forms: codes equal to the zero points give y = 0; codes one above them with
    unit scales give the row sums of x; a scale of 2^e scales y by 2^e exactly.
"""
import numpy as np

from oracle import w4_oracle as W
from synthetic import gen
from paper_2607_15865_gb300.w4 import pack_codes, pack_tiles


def test_packer_and_reader_agree_on_the_format():
    N, K = 37, 384
    codes = gen.uint4_codes("w4pin", "codes", (N, K))
    zeros = gen.uint4_codes("w4pin", "zeros", (N, K // 128))
    scales = gen.normal_bf16("w4pin", "scales", (N, K // 128), 0.02)
    buf = pack_tiles(pack_codes(codes), scales, zeros)
    assert buf.size == 3 * 3 * W.TILE_BYTES
    c, s, z = W.unpack_tiles(buf, N, K)
    assert (c == codes).all() and (s == scales).all() and (z == zeros).all()


def test_single_values_land_where_the_format_says():
    N, K = 20, 256
    codes = np.zeros((N, K), np.uint8)
    codes[19, 128 + 8 * 5 + 3] = 9  # tile row 1, group 1, row 3 of the tile, word 5, j = 3
    scales = np.zeros((N, 2), np.uint16)
    scales[17, 1] = 0x3F80  # 1.0: tile (1, 1), row 1
    zeros = np.zeros((N, 2), np.uint8)
    zeros[18, 0] = 7  # tile (1, 0), row 2
    buf = pack_tiles(pack_codes(codes), scales, zeros)
    rec = buf.reshape(4, W.TILE_BYTES)  # records (T, G) = (0,0), (0,1), (1,0), (1,1)
    word = rec[3, 64 * 3 + 4 * 5: 64 * 3 + 4 * 5 + 4].view("<u4")[0]
    assert int(word) == 9 << 20
    assert int(rec[3, 1024 + 2 * 1]) | (int(rec[3, 1024 + 2 * 1 + 1]) << 8) == 0x3F80
    assert int(rec[2, 1056 + 2]) == 7
    nonzero = np.flatnonzero(buf)
    assert len(nonzero) == 4  # the code, two scale bytes, the zero point
    c, s, z = W.unpack_tiles(buf, N, K)
    assert (c == codes).all() and (s == scales).all() and (z == zeros).all()


def test_gemv_matches_brute_force():
    N, K, M = 3, 256, 2
    codes = gen.uint4_codes("w4pin", "bf_codes", (N, K))
    zeros = gen.uint4_codes("w4pin", "bf_zeros", (N, K // 128))
    scales = gen.normal_bf16("w4pin", "bf_scales", (N, K // 128), 0.02)
    x = gen.normal_bf16("w4pin", "bf_x", (M, K), 1.0)
    xf = W.bf16_to_f64(x)
    sf = W.bf16_to_f64(scales)
    ref = np.zeros((M, N))
    for m in range(M):
        for n in range(N):
            t = 0.0
            for k in range(K):
                g = k // 128
                t += float(xf[m, k]) * (int(codes[n, k]) - int(zeros[n, g])) * float(sf[n, g])
            ref[m, n] = t
    got = W.gemv(codes, scales, zeros, x)
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_gemv_closed_forms():
    N, K, M = 5, 384, 3
    x = gen.normal_bf16("w4pin", "cf_x", (M, K), 1.0)
    xf = W.bf16_to_f64(x)
    zeros = gen.uint4_codes("w4pin", "cf_zeros", (N, K // 128)) % 15  # leave room for +1
    codes = np.repeat(zeros, 128, axis=1).astype(np.uint8)
    one = gen.f32_to_bf16_bits(np.ones((N, K // 128), np.float32))
    assert (W.gemv(codes, one, zeros, x) == 0).all()
    y1 = W.gemv(codes + 1, one, zeros, x)
    assert np.allclose(y1, np.repeat(xf.sum(axis=1, keepdims=True), N, axis=1), rtol=0, atol=1e-12)
    four = gen.f32_to_bf16_bits(np.full((N, K // 128), 4.0, np.float32))
    rnd = gen.uint4_codes("w4pin", "cf_codes", (N, K))
    assert (W.gemv(rnd, four, zeros, x) == 4 * W.gemv(rnd, one, zeros, x)).all()
