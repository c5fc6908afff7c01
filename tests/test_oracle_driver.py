"""Pins of the stage driver's oracle (Sections 4.1 and 4.5) against the plain definition.

The driver only reorders whole rows between stage calls, so the oracle of a prompt run
in segments must equal one prefill_kv of the whole prompt bit for bit, whatever the
segment length; and n decode steps (one token each, positions hist, hist+1, ...) must
equal one prefill_kv of the same n tokens (decode is prefill_kv with a chunk of one,
Section 4.4), row for row and cache slot for cache slot.
"""
import numpy as np
import pytest

from oracle import oracle as O
from synthetic import workloads as w
from synthetic.workloads import Shape

SHAPES = [Shape("drv_d64", 2, 4, 2, 64, 160, 1.0e4), Shape("drv_d128", 1, 6, 2, 128, 96, 1.0e6)]


@pytest.mark.parametrize("shape", SHAPES, ids=[s.name for s in SHAPES])
@pytest.mark.parametrize("hist", [0, 21])
@pytest.mark.parametrize("seg", [1, 7, 32, 500])
def test_segmented_prompt_equals_one_prefill_kv(shape, hist, seg):
    P = 60
    q, k, v = w.tokens(shape, "drv_prompt", P)
    kc, vc = w.cache(shape, "drv_prompt", hist, fill="random")
    rk, rv = kc.copy(), vc.copy()
    got = O.prompt(shape, q, k, v, hist, seg, kc, vc)
    ref = (O.prefill(shape, q, k, v, rk, rv) if hist == 0 else O.prefill_kv(shape, q, k, v, hist, rk, rv))
    assert (got == ref).all()
    assert (kc == rk).all() and (vc == rv).all()


@pytest.mark.parametrize("shape", SHAPES, ids=[s.name for s in SHAPES])
def test_decode_steps_equal_prefill_kv_of_the_same_tokens(shape):
    n, hist = 9, 40
    q, k, v = w.tokens(shape, "drv_dec", n)  # [B, n, H, D]
    kc, vc = w.cache(shape, "drv_dec", hist, fill="random")
    rk, rv = kc.copy(), vc.copy()
    step = lambda a: np.ascontiguousarray(a.transpose(1, 0, 2, 3)[:, :, None])  # [n, B, 1, H, D]
    got = O.decode_steps(shape, step(q), step(k), step(v), np.full(shape.batch, hist, np.int32), kc, vc)
    ref = O.prefill_kv(shape, q, k, v, hist, rk, rv)
    assert (got[:, :, 0].transpose(1, 0, 2, 3) == ref).all()
    assert (kc == rk).all() and (vc == rv).all()


def test_decode_steps_follow_each_sequence_own_length():
    shape = SHAPES[0]
    n = 4
    q, k, v = w.tokens(shape, "drv_mixed", n)
    hist = np.array([10, 73], np.int32)
    kc, vc = w.cache(shape, "drv_mixed", int(hist.max()), fill="random")
    rk, rv = kc.copy(), vc.copy()
    step = lambda a: np.ascontiguousarray(a.transpose(1, 0, 2, 3)[:, :, None])
    got = O.decode_steps(shape, step(q), step(k), step(v), hist, kc, vc)
    for t in range(n):
        ref = O.decode(shape, step(q)[t], step(k)[t], step(v)[t], hist + t, rk, rv)
        assert (got[t] == ref).all()
    assert (kc == rk).all() and (vc == rv).all()


def test_multi_token_decode_one_token_is_decode():
    shape = SHAPES[0]
    q, k, v = w.tokens(shape, "mtd1", 1)
    hist = np.array([12, 99], np.int32)
    kc, vc = w.cache(shape, "mtd1", int(hist.max()), fill="random")
    rk, rv = kc.copy(), vc.copy()
    got = O.decode_multi(shape, q, k, v, hist, kc, vc)
    ref = O.decode(shape, q, k, v, hist, rk, rv)
    assert (got == ref).all()
    assert (kc == rk).all() and (vc == rv).all()


def test_multi_token_decode_equals_decode_steps():
    """n new tokens at once = n single-token decode steps (each token sees the earlier new
    tokens, as they were appended by the earlier steps)."""
    shape = SHAPES[0]
    n = 5
    q, k, v = w.tokens(shape, "mtd2", n)
    hist = np.array([3, 70], np.int32)
    kc, vc = w.cache(shape, "mtd2", int(hist.max()), fill="random")
    rk, rv = kc.copy(), vc.copy()
    got = O.decode_multi(shape, q, k, v, hist, kc, vc)
    step = lambda a: np.ascontiguousarray(a.transpose(1, 0, 2, 3)[:, :, None])
    ref = O.decode_steps(shape, step(q), step(k), step(v), hist, rk, rv)
    assert (got == ref[:, :, 0].transpose(1, 0, 2, 3)).all()
    assert (kc == rk).all() and (vc == rv).all()
