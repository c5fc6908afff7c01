"""The seeded input generator: published test vectors, distribution, bf16 rounding."""
import numpy as np

from synthetic import gen
from synthetic import workloads as w


def test_splitmix64_published_vectors():
    # First outputs of splitmix64 from state 0 (Vigna's reference splitmix64.c).
    got = [int(x) for x in gen.splitmix64_stream(0, 0, 3)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_fnv1a64_published_vectors():
    assert gen.fnv1a64("") == 0xCBF29CE484222325
    assert gen.fnv1a64("a") == 0xAF63DC4C8601EC8C


def test_normal_moments_and_determinism():
    x = gen.normal_f64(gen.tensor_key("t", "x"), 400_001)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    assert (x == gen.normal_f64(gen.tensor_key("t", "x"), 400_001)).all()
    # a prefix of a stream does not depend on its length (counter based)
    assert (gen.normal_f64(gen.tensor_key("t", "x"), 1001)[:1000] == x[:1000]).all()
    assert not (gen.normal_f64(gen.tensor_key("t", "y"), 1000) == x[:1000]).any()


def test_bf16_round_to_nearest_even():
    xs = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -8 + 2 ** -20, -2.5, 0.0], np.float32)
    got = gen.f32_to_bf16_bits(xs)
    assert [hex(v) for v in got] == ["0x3f80", "0x3f80", "0x3f82", "0x3f81", "0xc020", "0x0"]
    assert (gen.bf16_bits_to_f32(got)[[0, 4]] == np.array([1.0, -2.5], np.float32)).all()


def test_workload_shapes():
    q, k, v = w.tokens(w.TINY, "chain", 28)
    assert q.shape == (1, 28, 4, 64) and k.shape == v.shape == (1, 28, 2, 64)
    kc, vc = w.cache(w.PREFILL_KV, "h", 1536)
    assert kc.shape == (1, 8, 2048, 128) and (kc[:, :, 1536:] == 0).all() and (kc[:, :, :1536] != 0).any()
    std = gen.bf16_bits_to_f32(q).std()
    assert abs(std - 1 / 8) < 0.01


def test_threaded_normal_equals_direct_definition():
    """The chunked, threaded evaluation equals Box-Muller applied directly to the stream."""
    key = gen.tensor_key("t", "direct")
    n = 3 * (1 << 20) + 7
    z = gen.splitmix64_stream(key, 0, 2 * ((n + 1) // 2)).reshape(-1, 2)
    u1 = ((z[:, 0] >> np.uint64(11)).astype(np.float64) + 1.0) / 2.0 ** 53
    u2 = (z[:, 1] >> np.uint64(11)).astype(np.float64) / 2.0 ** 53
    r = np.sqrt(-2.0 * np.log(u1))
    ref = np.stack([r * np.cos(2 * np.pi * u2), r * np.sin(2 * np.pi * u2)], 1).reshape(-1)[:n]
    assert (gen.normal_f64(key, n) == ref).all()
