"""GPU parity of decode (K1 + K3 + K4 through the C ABI) against the CPU oracle.

Covers the decode sweep (batch 1/4/16 x valid lengths 1024/4096/8191 over a
static maximum of 8192), mixed per-sequence lengths including 0 and max_len-1,
group sizes 1/7/16 and head_dim 64, the long-context point (32767 valid tokens),
and out-of-range lengths, which must set the device error word and leave that
sequence's cache and output untouched.  Slots past hist_len[b] hold NaN.
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


def run_decode(torch, shape, q, k, v, hist, kc, vc, out_init=None):
    from paper_2607_15865_gb300.attention import Attention
    attn = Attention.for_shape(shape)
    gk, gv = to_dev(kc), to_dev(vc)
    hl = torch.from_numpy(np.asarray(hist, np.int32)).cuda()
    out = to_dev(out_init) if out_init is not None else None
    out = attn.decode(to_dev(q), to_dev(k), to_dev(v), hl, gk, gv, out=out)
    torch.cuda.synchronize()
    flags = attn.device_error()
    res = to_host(out), to_host(gk), to_host(gv), flags
    attn.close()
    return res


def check_decode(torch, shape, tag, hist, rows=None):
    hist = np.asarray(hist, np.int32)
    q, k, v = w.tokens(shape, tag, 1)
    kc, vc = w.cache(shape, tag, int(hist.max()), fill="nan")
    for b in range(shape.batch):  # sequence b has hist[b] valid slots; the rest stays NaN
        kc[b, :, hist[b]:] = 0x7FC0
        vc[b, :, hist[b]:] = 0x7FC0
    out, gk, gv, flags = run_decode(torch, shape, q, k, v, hist, kc, vc)
    assert flags == 0
    rk, rv = kc.copy(), vc.copy()
    O.append(shape, k, v, hist, rk, rv)
    assert_cache(gk, gv, rk, rv, kc, vc, [(int(h), int(h) + 1) for h in hist], f"{tag} cache")
    if rows is None:
        rows = np.array([(b, 0, h) for b in range(shape.batch) for h in range(shape.n_q_heads)], np.int32)
    ref = O.attend_rows(shape, q, hist, rk, rv, rows)
    assert_out_close(out[rows[:, 0], rows[:, 1], rows[:, 2]], ref, tag)


SWEEP = [(b, h) for b in w.DECODE_BATCHES for h in w.DECODE_HISTS]


@pytest.mark.parametrize("batch,hist", SWEEP, ids=[f"b{b}_hist{h}" for b, h in SWEEP])
def test_decode_sweep(torch, batch, hist):
    shape = w.decode_shape(batch)
    rows = None
    if batch > 4:
        rng = np.random.default_rng(batch * 7 + hist)
        pick = [(b, 0, h) for b in (0, batch - 1) for h in range(shape.n_q_heads)]
        pick += [(int(rng.integers(batch)), 0, int(rng.integers(shape.n_q_heads))) for _ in range(32)]
        rows = np.array(pick, np.int32)
    check_decode(torch, shape, f"sweep_b{batch}_{hist}", [hist] * batch, rows)


def test_decode_mixed_lengths(torch):
    shape = Shape("mixed", 5, 32, 8, 128, 8192, 5.0e5)
    check_decode(torch, shape, "mixed", [0, 1, 127, 4097, 8191])


@pytest.mark.parametrize("shape,hist", [
    (Shape("g7", 2, 28, 4, 128, 1500, 1.0e6), [700, 1499]),
    (Shape("g1_d64", 3, 4, 4, 64, 900, 1.0e4), [3, 500, 899]),
    (Shape("g16", 1, 16, 1, 128, 2000, 1.0e4), [1999]),
    (Shape("g5_d64", 2, 10, 2, 64, 300, 1.0e4), [31, 32]),
], ids=["group7", "group1_d64", "group16", "group5_d64"])
def test_decode_group_sizes(torch, shape, hist):
    check_decode(torch, shape, shape.name, hist)


def test_decode_long_context(torch):
    shape = Shape("long_decode", 1, 40, 8, 128, 32768, 1.0e6)
    check_decode(torch, shape, "long_decode", [w.LONG_DECODE_HIST])


def test_decode_out_of_range_length_sets_error_and_skips(torch):
    shape = Shape("badlen", 3, 8, 2, 128, 256, 1.0e4)
    q, k, v = w.tokens(shape, "badlen", 1)
    kc, vc = w.cache(shape, "badlen", 200, fill="zero")
    sentinel = np.full(q.shape, 0x4049, np.uint16)  # 3.14 in bf16
    hist = [100, -1, 256]
    out, gk, gv, flags = run_decode(torch, shape, q, k, v, hist, kc, vc, out_init=sentinel)
    assert flags & 1, "an out-of-range hist_len must set ATTN_DEVERR_HIST_RANGE"
    for b in (1, 2):
        assert (out[b] == sentinel[b]).all(), "a skipped sequence's output must not be written"
        assert (gk[b] == kc[b]).all() and (gv[b] == vc[b]).all(), "a skipped sequence's cache must not change"
    rk, rv = kc.copy(), vc.copy()
    one = Shape("badlen1", 1, 8, 2, 128, 256, 1.0e4)
    r0k, r0v = rk[:1].copy(), rv[:1].copy()
    ref = O.decode(one, q[:1].copy(), k[:1].copy(), v[:1].copy(), np.array([100], np.int32), r0k, r0v)
    assert_out_close(out[:1], ref, "valid sequence next to invalid ones")


# More (sequence, kv head) items than half the SMs: the grid runs several waves of splits
# that claim what their items still have (split 0 of every item first).
MULTIWAVE = [
    ("b24_g4_lengths_0_to_4095", Shape("mw1", 24, 16, 4, 128, 4096, 1.0e4)),
    ("b16_g4_lengths_64_to_8191", Shape("mw2", 16, 32, 8, 128, 8192, 5.0e5)),
]


@pytest.mark.parametrize("name,shape", MULTIWAVE, ids=[m[0] for m in MULTIWAVE])
def test_decode_multiwave_mixed_lengths(torch, name, shape):
    rng = np.random.default_rng(len(name))
    lo = 0 if shape.max_len == 4096 else 64
    hist = rng.integers(lo, shape.max_len, size=shape.batch).astype(np.int32)
    hist[0], hist[-1] = lo, shape.max_len - 1
    pick = [(b, 0, h) for b in range(shape.batch) for h in (0, shape.n_q_heads - 1)]
    pick += [(int(rng.integers(shape.batch)), 0, int(rng.integers(shape.n_q_heads))) for _ in range(48)]
    check_decode(torch, shape, name, hist, np.array(pick, np.int32))


# One wave of splits whose items (sequence, kv head) fit as one thread-block cluster each
# merge through distributed shared memory, the others through global memory.  On a GB300
# (152 SMs, one 211 KB CTA per SM: 7 clusters of 16 CTAs fit at once, 8 of 12, 15 of 8, 23 of
# 6, 28 of 5, 36 of 4, 46 of 3, 76 of 2) these batches (G = 8 or 16, one kv head, so items =
# batch) take splits = min(16, 152 / items, tiles), lowered to a cluster size that fits when
# the cache holds at most 64 tiles: clusters of 16, 16 (exactly 7), 12, 8, 6, 5, 3 and 2, and
# the global merge at 16 and 4 splits over 65 tiles.  Lengths are mixed, so some items have
# fewer tiles than splits and short ones a single tile.
ONEWAVE_MERGES = [
    ("b1_g8_cluster16", Shape("ow1", 1, 8, 1, 128, 2048, 1.0e4)),
    ("b7_g8_cluster16", Shape("ow7", 7, 8, 1, 128, 2048, 1.0e4)),
    ("b8_g8_cluster12", Shape("ow8", 8, 8, 1, 128, 2048, 1.0e4)),
    ("b8_g8_global16", Shape("ow8g", 8, 8, 1, 128, 8320, 1.0e4)),
    ("b10_g8_cluster8", Shape("ow10", 10, 8, 1, 128, 1024, 1.0e4)),
    ("b22_g8_cluster6", Shape("ow22", 22, 8, 1, 128, 2048, 1.0e4)),
    ("b28_g8_cluster5", Shape("ow28", 28, 8, 1, 128, 2048, 1.0e4)),
    ("b38_g8_cluster3", Shape("ow38", 38, 8, 1, 128, 2048, 1.0e4)),
    ("b38_g8_global4", Shape("ow38g", 38, 8, 1, 128, 8320, 1.0e4)),
    ("b76_g8_cluster2", Shape("ow76", 76, 8, 1, 128, 512, 1.0e4)),
    ("b5_g16_cluster16", Shape("ow5g16", 5, 16, 1, 128, 2048, 1.0e4)),
]


@pytest.mark.parametrize("name,shape", ONEWAVE_MERGES, ids=[m[0] for m in ONEWAVE_MERGES])
def test_decode_one_wave_merges(torch, name, shape):
    rng = np.random.default_rng(len(name) * 31 + shape.batch)
    hist = rng.integers(0, shape.max_len, size=shape.batch).astype(np.int32)
    hist[0] = shape.max_len - 1
    if shape.batch > 2:
        hist[1], hist[2] = 0, 127  # a single key, and a single full tile
    check_decode(torch, shape, name, hist)


REPEATED = [
    # several waves of splits (160 items)
    ("multiwave", Shape("mwrep", 20, 16, 8, 128, 2048, 1.0e4)),
    # one wave (16 items x 9 splits): single-tile sequences next to ones with more tiles
    # than splits, so that a call whose item needs no counter precedes one that does
    ("onewave", Shape("owrep", 2, 16, 8, 128, 4096, 1.0e4)),
]


@pytest.mark.parametrize("name,shape", REPEATED, ids=[r[0] for r in REPEATED])
def test_decode_repeated_calls_leave_counters_clean(torch, name, shape):
    """Four calls on one context with different length mixes: the per-item counters
    (claims, slots, visits, done words) must be back at zero after every launch."""
    from paper_2607_15865_gb300.attention import Attention
    attn = Attention.for_shape(shape)
    rng = np.random.default_rng(5)
    for i in range(4):
        hist = rng.integers(0, shape.max_len, size=shape.batch).astype(np.int32)
        if i == 2:
            hist[:] = shape.max_len - 1
        if i % 2 == 0:
            hist[0] = 17  # one key tile
        else:
            hist[0] = shape.max_len - 1 - i
        q, k, v = w.tokens(shape, f"mwrep_{i}", 1)
        kc, vc = w.cache(shape, f"mwrep_{i}", int(hist.max()), fill="random")
        hl = torch.from_numpy(hist).cuda()
        out = to_host(attn.decode(to_dev(q), to_dev(k), to_dev(v), hl, to_dev(kc), to_dev(vc)))
        rk, rv = kc.copy(), vc.copy()
        ref = O.decode(shape, q, k, v, hist, rk, rv)
        assert_out_close(out, ref, f"{name}: call {i}")
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    attn.close()


def test_decode_chain_reuses_merge_state(torch):
    """Consecutive decode steps on one context and one cache: each step appends its
    token and attends to the previous steps' tokens; tile boundaries (128, 256) and
    splits without keys are crossed on the way.  Checks that nothing a step leaves
    behind on the device (merge counters, partials) changes the next step."""
    from paper_2607_15865_gb300.attention import Attention
    shape = Shape("chain", 2, 16, 8, 128, 1024, 1.0e4)
    hist0 = np.array([126, 254], np.int32)
    steps = 4
    kc, vc = w.cache(shape, "chain", int(hist0.max()), fill="random")
    attn = Attention.for_shape(shape)
    gk, gv = to_dev(kc), to_dev(vc)
    rk, rv = kc.copy(), vc.copy()
    for i in range(steps):
        hist = hist0 + i
        q, k, v = w.tokens(shape, f"chain_{i}", 1)
        hl = torch.from_numpy(hist).cuda()
        out = to_host(attn.decode(to_dev(q), to_dev(k), to_dev(v), hl, gk, gv))
        ref = O.decode(shape, q, k, v, hist, rk, rv)  # appends to rk, rv in place
        assert_out_close(out, ref, f"chain step {i}")
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    assert_cache(to_host(gk), to_host(gv), rk, rv, kc, vc,
                 [(int(h), int(h) + steps) for h in hist0], "chain cache")
    attn.close()
