"""Pins of the W4BF16 oracle (oracle/w4_oracle.py): each takes the oracle module, so that the
same pins run against the real oracle (tests/test_w4_oracle.py) and against copies with a
planted mistake (tests/test_w4_oracle_mutants.py).  None of them is the oracle's own code:

  * format: the oracle's writer and reader round-trip every code, scale and zero point of
    a matrix whose rows do not fill the last tile, and single values written by the oracle
    land at the byte and bit the documented format names (read back here by hand);
  * brute force: y[m, n] = sum_k x[m, k] (q[n, k] - z[n, k // 128]) s[n, k // 128] and RMSNorm
    written as plain Python loops on tiny cases;
  * closed forms: codes equal to the zero points give y = 0; codes one above them with
    unit scales give the row sums of x; a scale of 2^e scales y by 2^e exactly; known bf16
    values; rounding ties; a constant row normalises to +-gamma;
  * the block around attention: a zero o_proj returns x; q = 0 with o_proj = I returns x plus
    the mean of the visible v rows, and the appended v is the v projection of RMSNorm(x).
"""
import numpy as np

from synthetic import gen


def pin_writer_and_reader_agree_on_the_format(W):
    N, K = 37, 384
    codes = gen.uint4_codes("w4pin", "codes", (N, K))
    zeros = gen.uint4_codes("w4pin", "zeros", (N, K // 128))
    scales = gen.normal_bf16("w4pin", "scales", (N, K // 128), 0.02)
    buf = W.write_tiles(codes, scales, zeros)
    assert buf.size == 3 * 3 * W.TILE_BYTES
    c, s, z = W.unpack_tiles(buf, N, K)
    assert (c == codes).all() and (s == scales).all() and (z == zeros).all()


def pin_single_values_land_where_the_format_says(W):
    N, K = 20, 256
    codes = np.zeros((N, K), np.uint8)
    codes[19, 128 + 8 * 5 + 3] = 9  # tile row 1, group 1, row 3 of the tile, word 5, j = 3
    scales = np.zeros((N, 2), np.uint16)
    scales[17, 1] = 0x3F80  # 1.0: tile (1, 1), row 1
    zeros = np.zeros((N, 2), np.uint8)
    zeros[18, 0] = 7  # tile (1, 0), row 2
    buf = W.write_tiles(codes, scales, zeros)
    rec = buf.reshape(4, W.TILE_BYTES)  # records (T, G) = (0,0), (0,1), (1,0), (1,1)
    word = rec[3, 64 * 3 + 4 * 5: 64 * 3 + 4 * 5 + 4].view("<u4")[0]
    assert int(word) == 9 << 20
    assert int(rec[3, 1024 + 2 * 1]) | (int(rec[3, 1024 + 2 * 1 + 1]) << 8) == 0x3F80
    assert int(rec[2, 1056 + 2]) == 7
    nonzero = np.flatnonzero(buf)
    assert len(nonzero) == 4  # the code, two scale bytes, the zero point
    c, s, z = W.unpack_tiles(buf, N, K)
    assert (c == codes).all() and (s == scales).all() and (z == zeros).all()


def pin_gemv_matches_brute_force(W):
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


def pin_gemv_closed_forms(W):
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


# ----------------------------------------------------------------------------- the block around attention

def pin_bf16_rounding_is_nearest_even(W):
    assert (W.bf16_to_f64(np.array([0x3F80, 0xC020, 0x0000, 0x3C00], np.uint16)) == [1.0, -2.5, 0.0, 2.0 ** -7]).all()
    one = 1.0
    cases = {one: 0x3F80, one + 2.0 ** -8: 0x3F80, one + 3 * 2.0 ** -8: 0x3F82, one + 2.0 ** -8 + 2.0 ** -30: 0x3F81,
             -2.5: 0xC020, 0.0: 0x0000}
    for v, want in cases.items():
        got = int(W.to_bf16_bits(np.array([v]))[0])
        assert got == want, (v, hex(got))
    # values exactly representable in float32: the input generator's own float32 -> bf16 rounding
    f = (gen.normal_bf16("w4pin", "rnd_hi", (4096,), 1.0).astype(np.uint32) << np.uint32(16)).view(np.float32)
    f = f + (gen.uint4_codes("w4pin", "rnd_lo", (4096,)).astype(np.float32) - 7.5) * np.abs(f) * 2.0 ** -10
    assert (W.to_bf16_bits(f.astype(np.float64)) == gen.f32_to_bf16_bits(f)).all()


def pin_rmsnorm_brute_force_and_closed_forms(W):
    M, K = 2, 256
    x = gen.normal_bf16("w4pin", "rms_x", (M, K), 1.0)
    g = gen.normal_bf16("w4pin", "rms_g", (K,), 0.3)
    xf, gf = W.bf16_to_f64(x), W.bf16_to_f64(g)
    got = W.rmsnorm(x, g, 0.25)
    for m in range(M):
        ss = 0.0
        for k in range(K):
            ss += float(xf[m, k]) ** 2
        r = 1.0 / (ss / K + 0.25) ** 0.5
        want = W.to_bf16_bits(np.array([float(xf[m, k]) * r * float(gf[k]) for k in range(K)]))
        assert (got[m] == want).all()
    # a constant row c: x * r = sign(c) exactly (eps = 0), so the output is +-gamma
    c = gen.f32_to_bf16_bits(np.array([[-3.0] * K, [0.375] * K], np.float32))
    out = W.rmsnorm(c, g, 0.0)
    assert (out[0] == (g ^ np.uint16(0x8000))).all() and (out[1] == g).all()
    # scaling x by a power of two changes nothing (eps = 0)
    x4 = gen.f32_to_bf16_bits((W.bf16_to_f64(x) * 4.0).astype(np.float32))
    assert (W.rmsnorm(x4, g, 0.0) == W.rmsnorm(x, g, 0.0)).all()


def _layer_case(shape, tag, q_zero=False, wo_kind="random"):
    """Inputs of one decode-layer step for the pins: (x, gamma, wqkv, wo, hist, caches)."""
    from synthetic import workloads as w
    D, hq, hkv = shape.head_dim, shape.n_q_heads, shape.n_kv_heads
    qd, kd, hidden = hq * D, hkv * D, hq * D
    B = shape.batch
    x = gen.normal_bf16("w4pin", f"{tag}_x", (B, hidden), 1.0)
    gamma = gen.normal_bf16("w4pin", f"{tag}_g", (hidden,), 1.0)
    zq = gen.uint4_codes("w4pin", f"{tag}_zq", (qd + 2 * kd, hidden // 128)) % 15
    cq = gen.uint4_codes("w4pin", f"{tag}_cq", (qd + 2 * kd, hidden))
    if q_zero:
        cq[:qd] = np.repeat(zq[:qd], 128, axis=1)
    sq = gen.normal_bf16("w4pin", f"{tag}_sq", (qd + 2 * kd, hidden // 128), 0.02) & np.uint16(0x7FFF)
    zo = gen.uint4_codes("w4pin", f"{tag}_zo", (hidden, qd // 128)) % 15
    so = gen.normal_bf16("w4pin", f"{tag}_so", (hidden, qd // 128), 0.02) & np.uint16(0x7FFF)
    if wo_kind == "zero":
        co = np.repeat(zo, 128, axis=1)
    elif wo_kind == "identity":
        co = np.repeat(zo, 128, axis=1)
        co[np.arange(hidden), np.arange(hidden)] += 1
        so = gen.f32_to_bf16_bits(np.ones((hidden, qd // 128), np.float32))
    else:
        co = gen.uint4_codes("w4pin", f"{tag}_co", (hidden, qd))
    hist = np.array([37 + 50 * b for b in range(B)], np.int32)
    kc, vc = w.cache(shape, f"{tag}_cache", int(hist.max()), fill="random")
    return x, gamma, (cq, sq, zq), (co, so, zo), hist, kc, vc


def pin_decode_layer_residual_only_when_o_proj_is_zero(W):
    from synthetic.workloads import Shape
    shape = Shape("w4layer_a", 2, 4, 2, 64, 256, 1.0e4)
    x, gamma, wqkv, wo, hist, kc, vc = _layer_case(shape, "lz", wo_kind="zero")
    h = W.decode_layer(shape, x, gamma, 1e-6, wqkv, wo, hist, kc, vc)
    assert (h == x).all()


def pin_decode_layer_with_q_zero_and_identity_o_proj_averages_v(W):
    """q = 0 makes every score equal, so attention returns the plain mean of the visible v rows
    (the new one included); with o_proj = I the block returns x + that mean."""
    from synthetic.workloads import Shape
    shape = Shape("w4layer_b", 2, 4, 2, 64, 256, 1.0e4)
    x, gamma, wqkv, wo, hist, kc, vc = _layer_case(shape, "lq", q_zero=True, wo_kind="identity")
    h = W.decode_layer(shape, x, gamma, 1e-6, wqkv, wo, hist, kc, vc)
    G, D = shape.n_q_heads // shape.n_kv_heads, shape.head_dim
    qd, kd = shape.n_q_heads * D, shape.n_kv_heads * D
    wv = tuple(a[qd + kd:] for a in wqkv)
    v_new = W.to_bf16_bits(W.gemv(*wv, W.rmsnorm(x, gamma, 1e-6))).reshape(shape.batch, shape.n_kv_heads, D)
    for b in range(shape.batch):
        assert (vc[b, :, hist[b]] == v_new[b]).all()
        o = np.concatenate([W.bf16_to_f64(vc[b, hq // G, :hist[b] + 1]).mean(axis=0) for hq in range(shape.n_q_heads)])
        want = W.to_bf16_bits(W.bf16_to_f64(x[b]) + W.bf16_to_f64(W.to_bf16_bits(o)))
        assert (h[b] == want).all()

def pin_gemm_rounds_each_weight_once(W):
    """The prefill-side reading: W_bf16 = bf16((q - z) s).  With power-of-two scales every
    (q - z) s is exact, so the GEMM equals the exact product; with other scales it equals
    Python loops over the rounded weights."""
    T, N, K = 3, 5, 256
    x = gen.normal_bf16("w4pin", "gm_x", (T, K), 1.0)
    codes = gen.uint4_codes("w4pin", "gm_c", (N, K))
    zeros = gen.uint4_codes("w4pin", "gm_z", (N, K // 128))
    p2 = gen.f32_to_bf16_bits(np.array([[2.0 ** -(5 + (n + g) % 4) for g in range(K // 128)] for n in range(N)],
                                       np.float32))
    assert (W.gemm_bf16w(codes, p2, zeros, x) == W.gemv(codes, p2, zeros, x)).all()
    s = gen.normal_bf16("w4pin", "gm_s", (N, K // 128), 0.02)
    wb = W.dequant_bf16(codes, s, zeros)
    sf = W.bf16_to_f64(s)
    for n in range(N):
        for k in range(0, K, 37):
            v = (int(codes[n, k]) - int(zeros[n, k // 128])) * float(sf[n, k // 128])
            assert int(wb[n, k]) == int(W.to_bf16_bits(np.array([v]))[0])
    ref = np.zeros((T, N))
    xf, wf = W.bf16_to_f64(x), W.bf16_to_f64(wb)
    for t in range(T):
        for n in range(N):
            ref[t, n] = sum(float(xf[t, k]) * float(wf[n, k]) for k in range(K))
    assert np.allclose(W.gemm_bf16w(codes, s, zeros, x), ref, rtol=1e-12, atol=1e-12)


def _prefill_case(shape, S, tag, pow2_scales=False, q_zero=False, wo_kind="random"):
    """Inputs of one prefill-block chunk for the pins: (x [B, S, hidden], gamma, wqkv, wo)."""
    D, hq, hkv = shape.head_dim, shape.n_q_heads, shape.n_kv_heads
    qd, kd, hidden = hq * D, hkv * D, hq * D
    x = gen.normal_bf16("w4pin", f"{tag}_x", (shape.batch, S, hidden), 1.0)
    gamma = gen.normal_bf16("w4pin", f"{tag}_g", (hidden,), 1.0)

    def scales(name, rows, groups):
        if pow2_scales:  # every (q - z) s exact in bf16: the GEMM reading equals the exact product
            e = gen.uint4_codes("w4pin", f"{tag}_{name}e", (rows, groups)) % 4
            return gen.f32_to_bf16_bits((2.0 ** -(5.0 + e)).astype(np.float32))
        return gen.normal_bf16("w4pin", f"{tag}_{name}", (rows, groups), 0.02) & np.uint16(0x7FFF)

    zq = gen.uint4_codes("w4pin", f"{tag}_zq", (qd + 2 * kd, hidden // 128)) % 15
    cq = gen.uint4_codes("w4pin", f"{tag}_cq", (qd + 2 * kd, hidden))
    if q_zero:
        cq[:qd] = np.repeat(zq[:qd], 128, axis=1)
    sq = scales("sq", qd + 2 * kd, hidden // 128)
    zo = gen.uint4_codes("w4pin", f"{tag}_zo", (hidden, qd // 128)) % 15
    so = scales("so", hidden, qd // 128)
    if wo_kind == "zero":
        co = np.repeat(zo, 128, axis=1)
    elif wo_kind == "identity":
        co = np.repeat(zo, 128, axis=1)
        co[np.arange(hidden), np.arange(hidden)] += 1
        so = gen.f32_to_bf16_bits(np.ones((hidden, qd // 128), np.float32))
    else:
        co = gen.uint4_codes("w4pin", f"{tag}_co", (hidden, qd))
    return x, gamma, (cq, sq, zq), (co, so, zo)


def pin_prefill_layer_equals_a_chain_of_decode_layers(W):
    """Section 4.1: a chunk through the prefill block equals its tokens one by one through the
    decode block (with weights exact in bf16 the two projection readings coincide): h and the
    caches bit for bit."""
    from synthetic import workloads as w
    from synthetic.workloads import Shape
    shape = Shape("w4pre_a", 2, 4, 2, 64, 320, 1.0e4)
    S, hist = 9, 131
    x, gamma, wqkv, wo = _prefill_case(shape, S, "pc", pow2_scales=True)
    kc, vc = w.cache(shape, "pc_cache", hist, fill="random")
    kc2, vc2 = kc.copy(), vc.copy()
    h = W.prefill_layer(shape, x, gamma, 1e-6, wqkv, wo, hist, kc, vc)
    for t in range(S):
        ht = W.decode_layer(shape, x[:, t].copy(), gamma, 1e-6, wqkv, wo, np.full(shape.batch, hist + t, np.int32),
                            kc2, vc2)
        assert (h[:, t] == ht).all(), t
    assert (kc == kc2).all() and (vc == vc2).all()


def pin_prefill_layer_residual_only_when_o_proj_is_zero(W):
    from synthetic import workloads as w
    from synthetic.workloads import Shape
    shape = Shape("w4pre_b", 1, 4, 1, 128, 300, 1.0e4)
    x, gamma, wqkv, wo = _prefill_case(shape, 70, "pz", wo_kind="zero")
    kc, vc = w.cache(shape, "pz_cache", 0, fill="random")
    assert (W.prefill_layer(shape, x, gamma, 1e-6, wqkv, wo, 0, kc, vc) == x).all()


def pin_prefill_layer_with_q_zero_and_identity_o_proj_averages_v(W):
    """q = 0: token i of the chunk weighs its hist + i + 1 visible keys equally, so with
    o_proj = I the block returns x + the mean of those v rows (the chunk's own v rows being
    its v projection of RMSNorm(x))."""
    from synthetic import workloads as w
    from synthetic.workloads import Shape
    shape = Shape("w4pre_c", 2, 4, 2, 64, 256, 1.0e4)
    S, hist = 6, 40
    x, gamma, wqkv, wo = _prefill_case(shape, S, "pq", q_zero=True, wo_kind="identity")
    kc, vc = w.cache(shape, "pq_cache", hist, fill="random")
    h = W.prefill_layer(shape, x, gamma, 1e-6, wqkv, wo, hist, kc, vc)
    G, D = shape.n_q_heads // shape.n_kv_heads, shape.head_dim
    qd, kd = shape.n_q_heads * D, shape.n_kv_heads * D
    wv = tuple(a[qd + kd:] for a in wqkv)
    hidden = x.shape[-1]
    xn = W.rmsnorm(x.reshape(-1, hidden), gamma, 1e-6)
    v_new = W.to_bf16_bits(W.gemm_bf16w(*wv, xn)).reshape(shape.batch, S, shape.n_kv_heads, D)
    for b in range(shape.batch):
        for i in range(S):
            assert (vc[b, :, hist + i] == v_new[b, i]).all()
            o = np.concatenate([W.bf16_to_f64(vc[b, hq // G, :hist + i + 1]).mean(axis=0)
                                for hq in range(shape.n_q_heads)])
            want = W.to_bf16_bits(W.bf16_to_f64(x[b, i]) + W.bf16_to_f64(W.to_bf16_bits(o)))
            assert (h[b, i] == want).all(), (b, i)


ALL_PINS = [pin_gemm_rounds_each_weight_once, pin_writer_and_reader_agree_on_the_format, pin_single_values_land_where_the_format_says, pin_gemv_matches_brute_force, pin_gemv_closed_forms, pin_bf16_rounding_is_nearest_even, pin_rmsnorm_brute_force_and_closed_forms, pin_decode_layer_residual_only_when_o_proj_is_zero, pin_decode_layer_with_q_zero_and_identity_o_proj_averages_v,
            pin_prefill_layer_equals_a_chain_of_decode_layers, pin_prefill_layer_residual_only_when_o_proj_is_zero,
            pin_prefill_layer_with_q_zero_and_identity_o_proj_averages_v]
