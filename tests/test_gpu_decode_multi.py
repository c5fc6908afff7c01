"""GPU parity of the multi-token decode (attn_decode_multi): n new tokens per sequence,
per-sequence lengths on the device, token i attending causally to slots [0, hist + i].

Compared with the oracle of the same stage (for each sequence, prefill_kv of its n
tokens over its own history; pinned in tests/test_oracle_driver.py to n single-token
decode steps), on group sizes and token counts that fill 8 or 16 MMA columns or several
groups of 16 columns (up to 16 heads x 16 tokens, and a ragged last group), new
tokens that straddle a key tile, an empty history, the long-context shape, lengths
that run past max_len, and the argument checks.
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


CASES = [
    ("g5_three_tokens", Shape("mt1", 2, 40, 8, 128, 2048, 1.0e6), [100, 1000], 3),
    ("g4_four_tokens_straddling_tiles", Shape("mt2", 2, 32, 8, 128, 1024, 5.0e5), [126, 255], 4),
    ("g2_two_tokens_empty_history", Shape("mt3", 2, 4, 2, 128, 256, 1.0e4), [0, 5], 2),
    ("g1_sixteen_tokens", Shape("mt4", 1, 2, 2, 128, 600, 1.0e4), [300], 16),
    ("g8_two_tokens_batch3", Shape("mt5", 3, 16, 2, 128, 512, 1.0e4), [7, 130, 400], 2),
    # more than 16 (query head, token) columns: groups of 16 columns on sibling CTAs
    ("g4_eight_tokens_2_groups", Shape("mt6", 2, 32, 8, 128, 2048, 5.0e5), [100, 1500], 8),
    ("g8_eight_tokens_4_groups", Shape("mt7", 2, 64, 8, 128, 1024, 1.0e6), [200, 900], 8),
    ("g16_sixteen_tokens_16_groups", Shape("mt8", 1, 16, 1, 128, 512, 1.0e4), [250], 16),
    ("g5_seven_tokens_ragged_group", Shape("mt9", 1, 40, 8, 128, 4096, 1.0e6), [4080], 7),
    # head_dim 64: the tokens as decode steps in order
    ("d64_g2_five_tokens", Shape("mt10", 3, 4, 2, 64, 512, 1.0e4), [0, 77, 400], 5),
    ("d64_g4_two_tokens_tiny", Shape("mt11", 1, 4, 1, 64, 32, 1.0e4), [24], 2),
]


def run_gpu(torch, shape, hist, n, fill="nan"):
    from paper_2607_15865_gb300.attention import Attention
    attn = Attention.for_shape(shape)
    q, k, v = w.tokens(shape, "mt", n)
    kc, vc = w.cache(shape, "mt", int(max(hist)), fill=fill)
    hl = np.asarray(hist, np.int32)
    gk, gv = to_dev(kc), to_dev(vc)
    out = attn.decode_multi(to_dev(q), to_dev(k), to_dev(v), torch.from_numpy(hl).cuda(), gk, gv)
    torch.cuda.synchronize()
    flags = attn.device_error()
    res = to_host(out), to_host(gk), to_host(gv), flags
    attn.close()
    return (q, k, v, kc, vc, hl), res


@pytest.mark.parametrize("name,shape,hist,n", CASES, ids=[c[0] for c in CASES])
def test_multi_token_decode_matches_oracle(torch, name, shape, hist, n):
    # history slots past each sequence's own length hold NaN in the shared fill: only
    # slots [0, hist[b]) may be read (the longest sequence's history is random data)
    (q, k, v, kc, vc, hl), (out, gk, gv, flags) = run_gpu(torch, shape, hist, n, fill="random")
    assert flags == 0
    rk, rv = kc.copy(), vc.copy()
    ref = O.decode_multi(shape, q, k, v, hl, rk, rv)
    assert_out_close(out, ref, f"{name} out")
    assert_cache(gk, gv, rk, rv, kc, vc, [(int(h), int(h) + n) for h in hl], f"{name} cache")


def test_multi_token_decode_long_context(torch):
    shape = w.LONG
    hist, n = [32765 - 3], 3
    (q, k, v, kc, vc, hl), (out, gk, gv, flags) = run_gpu(torch, shape, hist, n)
    assert flags == 0
    rk, rv = kc.copy(), vc.copy()
    ref = O.decode_multi(shape, q, k, v, hl, rk, rv)
    assert_out_close(out, ref, "long context out")
    assert_cache(gk, gv, rk, rv, kc, vc, [(hist[0], hist[0] + n)], "long context cache")


def test_one_new_token_is_attn_decode(torch):
    from paper_2607_15865_gb300.attention import Attention
    shape = Shape("mt_one", 2, 8, 2, 128, 512, 1.0e4)
    attn = Attention.for_shape(shape)
    q, k, v = w.tokens(shape, "mt_one", 1)
    kc, vc = w.cache(shape, "mt_one", 300, fill="random")
    hl = torch.from_numpy(np.array([17, 300], np.int32)).cuda()
    k1, v1, k2, v2 = to_dev(kc), to_dev(vc), to_dev(kc), to_dev(vc)
    a = attn.decode_multi(to_dev(q), to_dev(k), to_dev(v), hl, k1, v1)
    b = attn.decode(to_dev(q), to_dev(k), to_dev(v), hl, k2, v2)
    torch.cuda.synchronize()
    assert (to_host(a) == to_host(b)).all()
    assert (to_host(k1) == to_host(k2)).all() and (to_host(v1) == to_host(v2)).all()
    attn.close()


def test_multi_token_decode_past_max_len_flags_and_skips(torch):
    from paper_2607_15865_gb300 import _lib
    shape = Shape("mt_edge", 2, 8, 2, 128, 256, 1.0e4)
    n = 3
    hist = [254, 40]  # sequence 0 needs slots 254..256: out of range
    (q, k, v, kc, vc, hl), (out, gk, gv, flags) = run_gpu(torch, shape, hist, n, fill="random")
    assert flags & _lib.DEVERR_HIST_RANGE
    assert (gk[0] == kc[0]).all() and (gv[0] == vc[0]).all(), "skipped sequence's cache changed"
    import dataclasses
    one = dataclasses.replace(shape, batch=1)
    rk, rv = kc[1:].copy(), vc[1:].copy()
    ref = O.decode_multi(one, q[1:], k[1:], v[1:], hl[1:], rk, rv)
    assert_out_close(out[1:], ref, "in-range sequence")


def test_multi_token_decode_rejects_bad_shapes(torch):
    from paper_2607_15865_gb300 import _lib
    from paper_2607_15865_gb300.attention import Attention
    for shape, n in ((Shape("mt_bad1", 1, 40, 8, 128, 256, 1.0e4), 17),  # more than 16 new tokens
                     (Shape("mt_bad2", 1, 4, 2, 64, 16, 1.0e4), 17)):     # head_dim 64, more than max_len
        attn = Attention.for_shape(shape)
        q, k, v = (to_dev(a) for a in w.tokens(shape, "bad", n))
        kc, vc = (to_dev(a) for a in w.cache(shape, "bad", 0))
        hl = torch.zeros(1, dtype=torch.int32, device="cuda")
        with pytest.raises(_lib.AttnError) as e:
            attn.decode_multi(q, k, v, hl, kc, vc)
        assert e.value.code == _lib.ATTN_EINVAL
        attn.close()
