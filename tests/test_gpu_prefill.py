"""GPU parity of prefill and prefill_kv (K1 + K2 through the C ABI) against the CPU oracle.

Small shapes are compared row for row; the full-size workloads (7B-class prefill,
prefill_kv 512 over 1536, long context 4096 and 4096 over 28672) are compared on
sampled rows the oracle computes one by one, plus properties that hold for every
row (finite; each output element lies within the range of the values it averages).
Cache slots past hist+chunk are filled with NaN, so any read of them would show.
"""
import numpy as np
import pytest

from oracle import oracle as O
from synthetic import workloads as w
from synthetic.workloads import Shape
from tests.gpu_util import assert_cache, assert_out_close, f32, to_dev, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as t
    assert t.cuda.is_available(), "GPU tests need a CUDA device"
    import __graft_entry__
    __graft_entry__.build()
    return t


def gpu_stage(torch, shape, q, k, v, hist, kc, vc, use_prefill_entry=False):
    from paper_2607_15865_gb300.attention import Attention
    attn = Attention.for_shape(shape)
    gk, gv = to_dev(kc), to_dev(vc)
    if use_prefill_entry:
        out = attn.prefill(to_dev(q), to_dev(k), to_dev(v), gk, gv)
    else:
        out = attn.prefill_kv(to_dev(q), to_dev(k), to_dev(v), hist, gk, gv)
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    res = to_host(out), to_host(gk), to_host(gv)
    attn.close()
    return res


SMALL = [
    ("ragged_hist77_chunk200", Shape("r1", 1, 4, 2, 128, 512, 1.0e4), 77, 200),
    ("single_token_prefill", Shape("r2", 1, 4, 2, 128, 64, 1.0e4), 0, 1),
    ("mha_d64_batch2", Shape("r3", 2, 3, 3, 64, 400, 1.0e4), 130, 131),
    ("gqa7_prefill_3tiles", Shape("r4", 1, 14, 2, 128, 700, 1.0e6), 0, 300),
    ("batch3_hist256", Shape("r5", 3, 8, 2, 128, 600, 5.0e5), 256, 257),
    ("cache_full_to_max_len", Shape("r6", 1, 4, 1, 128, 384, 1.0e4), 128, 256),
    ("d64_hist1000", Shape("r7", 1, 4, 2, 64, 1100, 1.0e4), 1000, 100),
    ("group16", Shape("r8", 1, 16, 1, 128, 300, 1.0e4), 40, 150),
    ("tile_aligned_128_over_128", Shape("r9", 1, 2, 1, 128, 256, 1.0e4), 128, 128),
]


@pytest.mark.parametrize("name,shape,hist,chunk", SMALL, ids=[c[0] for c in SMALL])
def test_small_shapes_match_oracle(torch, name, shape, hist, chunk):
    q, k, v = w.tokens(shape, "small", chunk)
    kc, vc = w.cache(shape, "small", hist, fill="nan")
    rk, rv = kc.copy(), vc.copy()
    ref = O.prefill_kv(shape, q, k, v, hist, rk, rv)
    out, gk, gv = gpu_stage(torch, shape, q, k, v, hist, kc, vc)
    assert_out_close(out, ref, name)
    assert_cache(gk, gv, rk, rv, kc, vc, [(hist, hist + chunk)] * shape.batch, name)


def test_prefill_equals_prefill_kv_without_history(torch):
    """Section 4.2: prefill is the with_history=False instance of one template."""
    shape = Shape("tmpl", 2, 8, 2, 128, 520, 1.0e6)
    q, k, v = w.tokens(shape, "tmpl", 333)
    kc, vc = w.cache(shape, "tmpl", 0, fill="nan")
    a = gpu_stage(torch, shape, q, k, v, 0, kc, vc, use_prefill_entry=True)
    b = gpu_stage(torch, shape, q, k, v, 0, kc, vc)
    for x, y in zip(a, b):
        assert (x == y).all()


def test_tiny_stage_chain(torch):
    """Section 4.1 scenario 2 on the tiny workload: prefill 16, prefill_kv 8 over 16, 4 decodes,
    against the oracle and against a single prefill over all 28 tokens."""
    from paper_2607_15865_gb300.attention import Attention
    s = w.TINY
    q, k, v = w.tokens(s, "chain", 28)
    kc, vc = w.cache(s, "chain", 0, fill="nan")
    rk, rv = kc.copy(), vc.copy()
    ref_full = O.prefill(s, q, k, v, rk, rv)
    attn = Attention.for_shape(s)
    gk, gv = to_dev(kc), to_dev(vc)
    outs = [attn.prefill(to_dev(q[:, :16].copy()), to_dev(k[:, :16].copy()), to_dev(v[:, :16].copy()), gk, gv),
            attn.prefill_kv(to_dev(q[:, 16:24].copy()), to_dev(k[:, 16:24].copy()), to_dev(v[:, 16:24].copy()), 16,
                            gk, gv)]
    for t in range(24, 28):
        hl = torch.full((s.batch,), t, dtype=torch.int32, device="cuda")
        outs.append(attn.decode(to_dev(q[:, t:t + 1].copy()), to_dev(k[:, t:t + 1].copy()),
                                to_dev(v[:, t:t + 1].copy()), hl, gk, gv))
    chain = np.concatenate([to_host(o) for o in outs], axis=1)
    ck, cv = to_host(gk), to_host(gv)
    gk2, gv2 = to_dev(kc), to_dev(vc)
    full = to_host(attn.prefill(to_dev(q), to_dev(k), to_dev(v), gk2, gv2))
    torch.cuda.synchronize()
    assert attn.device_error() == 0
    assert_out_close(chain, ref_full, "tiny chain vs oracle")
    assert_out_close(full, ref_full, "tiny full prefill vs oracle")
    assert_cache(ck, cv, rk, rv, kc, vc, [(0, 28)], "tiny chain cache")
    assert (ck == to_host(gk2)).all() and (cv == to_host(gv2)).all(), "the chain and one prefill must leave equal caches"


def sample_rows(shape, chunk, n_pos, heads="all", seed=1):
    rng = np.random.default_rng(seed)
    fixed = {0, 1, chunk - 1, chunk - 2, min(127, chunk - 1), min(128, chunk - 1), chunk // 2}
    pos = sorted(fixed | set(rng.integers(0, chunk, size=n_pos).tolist()))
    hs = range(shape.n_q_heads) if heads == "all" else sorted(set(rng.integers(0, shape.n_q_heads, heads).tolist()))
    return np.array([(b, i, h) for b in range(shape.batch) for i in pos for h in hs], np.int32)


def check_full_size(torch, shape, tag, hist, chunk, n_pos, heads="all"):
    q, k, v = w.tokens(shape, tag, chunk)
    kc, vc = w.cache(shape, tag, hist, fill="nan")
    out, gk, gv = gpu_stage(torch, shape, q, k, v, hist, kc, vc)
    rk, rv = kc.copy(), vc.copy()
    O.append(shape, k, v, hist, rk, rv)
    assert_cache(gk, gv, rk, rv, kc, vc, [(hist, hist + chunk)] * shape.batch, f"{tag} cache")
    rows = sample_rows(shape, chunk, n_pos, heads)
    ref = O.attend_rows(shape, q, hist, rk, rv, rows)
    got = out[rows[:, 0], rows[:, 1], rows[:, 2]]
    assert_out_close(got, ref, f"{tag} sampled rows")
    # every row: finite and inside the range of the values it averages (per kv head, per element)
    o = f32(out)
    assert np.isfinite(o).all()
    vmax = np.abs(f32(rv[:, :, :hist + chunk])).max(axis=2)  # [B,Hkv,D]
    lim = np.repeat(vmax, shape.group, axis=1)[:, None] * (1 + 2.0 ** -7)  # [B,1,Hq,D]
    assert (np.abs(o) <= lim).all(), f"{tag}: an output lies outside the convex hull bound"


def test_prefill_7b_full(torch):
    """7B-class prefill (28 query heads, 4 KV heads, D=128, theta 1e6, 512 tokens), every row."""
    s = w.PREFILL_7B
    q, k, v = w.tokens(s, "prefill", 512)
    kc, vc = w.cache(s, "prefill", 0, fill="nan")
    rk, rv = kc.copy(), vc.copy()
    ref = O.prefill(s, q, k, v, rk, rv)
    out, gk, gv = gpu_stage(torch, s, q, k, v, 0, kc, vc, use_prefill_entry=True)
    assert_out_close(out, ref, "prefill_7b")
    assert_cache(gk, gv, rk, rv, kc, vc, [(0, 512)], "prefill_7b cache")


def test_prefill_kv_512_over_1536(torch):
    check_full_size(torch, w.PREFILL_KV, "pkv", 1536, 512, n_pos=24)


def test_long_prefill_4096(torch):
    check_full_size(torch, w.LONG, "long_prefill", 0, w.LONG_PREFILL, n_pos=10, heads=12)


def test_long_prefill_kv_4096_over_28672(torch):
    check_full_size(torch, w.LONG, "long_pkv", w.LONG_PKV_HIST, w.LONG_PKV_CHUNK, n_pos=6, heads=10)


# A prefill_kv whose history is at least its chunk and whose K/V exceeds about 42 MB:
# flash_fwd then groups its work items in blocks of kv heads of one sequence (blocks of 2
# kv heads on the long-context shape, of 1 here) instead of by query-tile pair.
def test_kv_head_blocks_batch2_every_row(torch):
    """A ragged 333-token chunk over 79000 history tokens, two sequences, 4 kv heads of
    GQA 3 (40.6 MB of K/V per kv head: one kv head per block), every row."""
    check_every_row(torch, Shape("kvb_b2", 2, 12, 4, 128, 79400, 1.0e6), "kvb_b2", 79000, 333)


def check_every_row(torch, shape, tag, hist, chunk):
    """Every output row of a full-size stage against the oracle, run on all host cores."""
    q, k, v = w.tokens(shape, tag, chunk)
    kc, vc = w.cache(shape, tag, hist, fill="nan")
    out, gk, gv = gpu_stage(torch, shape, q, k, v, hist, kc, vc)
    rk, rv = kc.copy(), vc.copy()
    O.append(shape, k, v, hist, rk, rv)
    assert_cache(gk, gv, rk, rv, kc, vc, [(hist, hist + chunk)] * shape.batch, f"{tag} cache")
    rows = np.array([(b, i, h) for b in range(shape.batch) for i in range(chunk) for h in range(shape.n_q_heads)],
                    np.int32)
    ref = O.attend_rows_parallel(shape, q, hist, rk, rv, rows).reshape(out.shape)
    assert_out_close(out, ref, f"{tag} every row")


@pytest.mark.slow
def test_long_prefill_4096_every_row(torch):
    check_every_row(torch, w.LONG, "long_prefill_all", 0, w.LONG_PREFILL)


@pytest.mark.slow
def test_long_prefill_kv_4096_over_28672_every_row(torch):
    check_every_row(torch, w.LONG, "long_pkv_all", w.LONG_PKV_HIST, w.LONG_PKV_CHUNK)
