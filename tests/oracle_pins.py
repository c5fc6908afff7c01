"""Pins that tie the CPU oracle to facts other than itself.

Each ``pin_*`` function takes a loaded oracle library and raises AssertionError
when the oracle disagrees with the fact it checks.  ``test_oracle_pins.py`` runs
them on the oracle; ``test_oracle_mutants.py`` runs them on copies of the oracle
with a planted mistake and requires that some pin fails for every mistake.

Sources of truth used here (none of them is the oracle's own code):
  * closed forms of the rotary table (angle p*theta^(-2j/D) equals p when j=0 and
    equals 1 at p=100, j=D/4 for theta=1e4) and of RoPE (identity at position 0);
  * RoPE as multiplication of the complex number x_j + i x_{j+D/2} by
    exp(i p omega_j), evaluated by numpy in complex128;
  * invariants of rotations: norm preservation, inner products that depend only
    on the position difference;
  * causal scaled dot-product attention from torch's library routine
    (``scaled_dot_product_attention`` on CPU in float64) with an explicit mask
    and the kv heads repeated per group;
  * closed-form attention results: one key (output = its value), a zero query
    (output = mean of the visible values), two keys of which one scores zero
    (output = logistic blend);
  * causality (a row never depends on later tokens, always on its own token) and
    the paper's stage composition (Section 4.1: prefill over a prompt equals prefill
    on a prefix, prefill_kv on the rest, then token-by-token decode).
"""
from __future__ import annotations

import math

import numpy as np
import torch

from oracle import oracle as O
from synthetic import gen
from synthetic import workloads as w
from synthetic.workloads import Shape

f32 = gen.bf16_bits_to_f32
bf16 = gen.f32_to_bf16_bits


def _omega(shape_or_dim, theta):
    d = shape_or_dim
    j = np.arange(d // 2, dtype=np.float64)
    return theta ** (-2.0 * j / d)


def complex_rope(x_bf16, p, d, theta):
    """RoPE as complex multiplication: (x_j + i x_{j+D/2}) * exp(i p omega_j), float64."""
    x = f32(x_bf16).astype(np.float64)
    h = d // 2
    z = (x[..., :h] + 1j * x[..., h:]) * np.exp(1j * p * _omega(d, theta))
    return np.concatenate([z.real, z.imag], axis=-1)


def _close(a, b, rtol, atol, what):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    err = np.abs(a - b)
    lim = rtol * np.abs(b) + atol
    bad = err > lim
    assert not bad.any(), f"{what}: {bad.sum()} of {bad.size} outside tolerance, max err {err.max():.3e}"


# ---------------------------------------------------------------- RoPE pins


def pin_table_closed_forms(lib):
    c, s = O.rope_tables(160, 64, 1.0e4, lib)
    assert (c[0] == 1.0).all() and (s[0] == 0.0).all(), "position 0 must give cos=1, sin=0"
    for p in range(160):  # j = 0: omega = 1, angle = p
        assert c[p, 0] == np.float32(math.cos(p)) and s[p, 0] == np.float32(math.sin(p)), p
    # j = D/4 = 16: omega = 1e4^(-1/2) = 1/100, so position 100 has angle 1.
    assert abs(float(c[100, 16]) - math.cos(1.0)) <= 1e-7
    assert abs(float(s[100, 16]) - math.sin(1.0)) <= 1e-7
    # j = D/8 = 8: omega = 1e4^(-1/4) = 1/10, so position 10 has angle 1.
    assert abs(float(c[10, 8]) - math.cos(1.0)) <= 1e-7


def pin_rope_complex(lib):
    for d, theta, p in ((64, 1.0e4, 7), (128, 1.0e6, 4095), (128, 5.0e5, 32767), (64, 1.0e4, 1)):
        c, s = O.rope_tables(p + 1, d, theta, lib)
        x = gen.normal_bf16("pin", f"rope{d}/{p}", (d,), 1.0)
        y = O.rope_row(x, c[p], s[p], lib)
        ref = complex_rope(x, p, d, theta)
        mag = np.abs(f32(x)).max()
        _close(y, ref, 0.0, 1e-6 * mag, f"rope d={d} p={p}")


def pin_rope_identity_norm_relative(lib):
    d, theta = 128, 1.0e6
    c, s = O.rope_tables(600, d, theta, lib)
    x = gen.normal_bf16("pin", "rope/x", (d,), 1.0)
    k = gen.normal_bf16("pin", "rope/k", (d,), 1.0)
    assert (O.rope_row(x, c[0], s[0], lib) == f32(x)).all(), "RoPE at position 0 must be the identity"
    n0 = float(np.sum(f32(x).astype(np.float64) ** 2))
    for p in (1, 17, 333, 599):
        y = O.rope_row(x, c[p], s[p], lib).astype(np.float64)
        assert abs(float(np.sum(y * y)) - n0) <= 1e-5 * n0, f"norm not preserved at p={p}"
    scale = float(np.linalg.norm(f32(x)) * np.linalg.norm(f32(k)))
    for (p, pp, t) in ((5, 2, 100), (300, 10, 250), (40, 41, 500)):
        a = np.dot(O.rope_row(x, c[p], s[p], lib).astype(np.float64),
                   O.rope_row(k, c[pp], s[pp], lib).astype(np.float64))
        b = np.dot(O.rope_row(x, c[p + t], s[p + t], lib).astype(np.float64),
                   O.rope_row(k, c[pp + t], s[pp + t], lib).astype(np.float64))
        assert abs(a - b) <= 2e-5 * scale, f"inner product depends on absolute position ({p},{pp},{t})"


# ---------------------------------------------------------------- attention pins


def _sdpa_reference(shape: Shape, qhat, kc, vc, hist, chunk):
    """Causal GQA SDPA over cache slots [0, hist+chunk) with torch's CPU routine in float64."""
    B, Hq, Hkv, D, G = shape.batch, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.group
    n = hist + chunk
    q = torch.from_numpy(f32(qhat).astype(np.float64)).permute(0, 2, 1, 3)  # [B,Hq,S,D]
    k = torch.from_numpy(f32(kc[:, :, :n]).astype(np.float64)).repeat_interleave(G, dim=1)
    v = torch.from_numpy(f32(vc[:, :, :n]).astype(np.float64)).repeat_interleave(G, dim=1)
    i = torch.arange(chunk).unsqueeze(1)
    j = torch.arange(n).unsqueeze(0)
    mask = j <= hist + i
    o = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=mask)
    return o.permute(0, 2, 1, 3).numpy()  # [B,S,Hq,D]


def pin_attention_matches_sdpa(lib):
    for shape, hist, chunk in ((Shape("pinA", 2, 6, 2, 32, 48, 1.0e4), 11, 13),
                               (Shape("pinB", 1, 4, 4, 64, 40, 5.0e5), 0, 21),
                               (Shape("pinC", 1, 8, 2, 128, 300, 1.0e6), 257, 30)):
        q, k, v = w.tokens(shape, "sdpa", chunk)
        kc, vc = w.cache(shape, "sdpa", hist, fill="random")
        kc0 = kc.copy()
        out = O.prefill_kv(shape, q, k, v, hist, kc, vc, lib)
        c, s = O.rope_tables(shape.max_len, shape.head_dim, shape.rope_theta, lib)
        # the new cache slots: bf16 of the complex-form rotation of k, v unchanged
        for i in range(chunk):
            p = hist + i
            ref = complex_rope(k[:, i], p, shape.head_dim, shape.rope_theta)  # [B,Hkv,D]
            got = f32(kc[:, :, p])
            _close(got, ref, 2.0 ** -7, 1e-6, f"{shape.name} k cache slot {p}")
            assert (vc[:, :, p] == v[:, i]).all(), f"{shape.name}: v cache slot {p} must hold v"
        assert (kc[:, :, :hist] == kc0[:, :, :hist]).all(), "history slots must be untouched"
        # rotated queries, rounded to bf16
        qhat = np.empty_like(q)
        for b in range(shape.batch):
            for i in range(chunk):
                for h in range(shape.n_q_heads):
                    p = hist + i
                    qhat[b, i, h] = bf16(O.rope_row(q[b, i, h], c[p], s[p], lib))
        ref = _sdpa_reference(shape, qhat, kc, vc, hist, chunk)
        _close(f32(out), ref, 2.0 ** -7, 1e-6, f"{shape.name} attention vs SDPA")


def pin_single_key(lib):
    shape = Shape("pin1", 2, 6, 2, 64, 8, 1.0e4)
    q, k, v = w.tokens(shape, "one", 1)
    kc, vc = w.cache(shape, "one", 0)
    out = O.prefill(shape, q, k, v, kc, vc, lib)
    for h in range(shape.n_q_heads):
        assert (out[:, 0, h] == v[:, 0, h // shape.group]).all(), \
            f"one visible key: head {h} must return the value of kv head {h // shape.group}"


def pin_zero_query(lib):
    shape = Shape("pin0", 2, 4, 2, 64, 64, 1.0e4)
    hist, chunk = 19, 9
    _, k, v = w.tokens(shape, "zero", chunk)
    q = np.zeros((shape.batch, chunk, shape.n_q_heads, shape.head_dim), np.uint16)
    kc, vc = w.cache(shape, "zero", hist, fill="random")
    out = O.prefill_kv(shape, q, k, v, hist, kc, vc, lib)
    for b in range(shape.batch):
        for i in range(chunk):
            for h in range(shape.n_q_heads):
                g = h // shape.group
                mean = f32(vc[b, g, :hist + i + 1]).astype(np.float64).mean(axis=0)
                _close(f32(out[b, i, h]), mean, 2.0 ** -7, 1e-7, "zero query gives the mean of visible v")


def pin_two_key_logistic(lib):
    d, theta = 64, 1.0e4
    shape = Shape("pin2", 1, 1, 1, d, 4, theta)
    kk = gen.normal_bf16("pin", "two/k0", (d,), 1.0)
    target = 0.35 * f32(kk).astype(np.float64)
    h = d // 2
    z = (target[:h] + 1j * target[h:]) * np.exp(-1j * 1 * _omega(d, theta))  # inverse rotation to p=1
    q1 = bf16(np.concatenate([z.real, z.imag]).astype(np.float32))
    q = np.stack([gen.normal_bf16("pin", "two/q0", (d,), 1.0), q1]).reshape(1, 2, 1, d)
    k = np.stack([kk, np.zeros(d, np.uint16)]).reshape(1, 2, 1, d)
    v = gen.normal_bf16("pin", "two/v", (1, 2, 1, d), 1.0)
    kc, vc = w.cache(shape, "two", 0)
    out = O.prefill(shape, q, k, v, kc, vc, lib)
    qhat = bf16(complex_rope(q1, 1, d, theta).astype(np.float32))
    s0 = float(np.dot(f32(qhat).astype(np.float64), f32(kk).astype(np.float64))) / math.sqrt(d)
    assert 1.0 < s0 < 5.0
    sig = 1.0 / (1.0 + math.exp(-s0))
    ref = sig * f32(v[0, 0, 0]).astype(np.float64) + (1.0 - sig) * f32(v[0, 1, 0]).astype(np.float64)
    _close(f32(out[0, 1, 0]), ref, 2.0 ** -7, 1e-6, "two keys give a logistic blend")


def pin_causality(lib):
    shape = Shape("pinc", 1, 4, 2, 64, 16, 1.0e4)
    S, t = 10, 5
    q, k, v = w.tokens(shape, "causal", S)
    kc, vc = w.cache(shape, "causal", 0)
    base = O.prefill(shape, q, k, v, kc.copy(), vc.copy(), lib)
    k2, v2 = k.copy(), v.copy()
    k2[:, t:] = gen.normal_bf16("pin", "causal/k2", k2[:, t:].shape, shape.scale)
    v2[:, t:] = gen.normal_bf16("pin", "causal/v2", v2[:, t:].shape, shape.scale)
    pert = O.prefill(shape, q, k2, v2, kc.copy(), vc.copy(), lib)
    assert (pert[:, :t] == base[:, :t]).all(), "a row must not depend on later tokens"
    assert (pert[:, t] != base[:, t]).any(axis=-1).all(), "a row must depend on its own token"


def pin_stage_chain(lib):
    """Section 4.1: prefill(28) == prefill(16) + prefill_kv(8 over 16) + 4 decodes (tiny workload)."""
    s = w.TINY
    q, k, v = w.tokens(s, "chain", 28)
    kc_a, vc_a = w.cache(s, "chain", 0)
    out_a = O.prefill(s, q, k, v, kc_a, vc_a, lib)
    kc_b, vc_b = w.cache(s, "chain", 0)
    parts = [O.prefill(s, q[:, :16].copy(), k[:, :16].copy(), v[:, :16].copy(), kc_b, vc_b, lib),
             O.prefill_kv(s, q[:, 16:24].copy(), k[:, 16:24].copy(), v[:, 16:24].copy(), 16, kc_b, vc_b, lib)]
    for t in range(24, 28):
        parts.append(O.decode(s, q[:, t:t + 1].copy(), k[:, t:t + 1].copy(), v[:, t:t + 1].copy(),
                              np.full(s.batch, t, np.int32), kc_b, vc_b, lib))
    assert (kc_a == kc_b).all() and (vc_a == vc_b).all(), "stage chain must leave identical caches"
    assert (np.concatenate(parts, axis=1) == out_a).all(), "stage chain must give identical outputs"


def pin_in_place(lib):
    shape = Shape("pini", 2, 4, 2, 64, 64, 1.0e4)
    hist, chunk = 20, 12
    q, k, v = w.tokens(shape, "inplace", chunk)
    kc, vc = w.cache(shape, "inplace", hist, fill="nan")
    kc0, vc0 = kc.copy(), vc.copy()
    out = O.prefill_kv(shape, q, k, v, hist, kc, vc, lib)
    keep = np.ones(shape.max_len, bool)
    keep[hist:hist + chunk] = False
    assert (kc[:, :, keep] == kc0[:, :, keep]).all() and (vc[:, :, keep] == vc0[:, :, keep]).all()
    assert np.isfinite(f32(out)).all(), "slots past hist+chunk must never be read"


def pin_decode_mixed_lengths(lib):
    shape = Shape("pind", 3, 8, 2, 64, 40, 5.0e5)
    hist = np.array([5, 0, 39], np.int32)
    q, k, v = w.tokens(shape, "mixed", 1)
    kc, vc = w.cache(shape, "mixed", 40, fill="random")
    kc0, vc0 = kc.copy(), vc.copy()
    out = O.decode(shape, q, k, v, hist, kc, vc, lib)
    one = Shape("pind1", 1, 8, 2, 64, 40, 5.0e5)
    for b in range(3):
        kb, vb = kc0[b:b + 1].copy(), vc0[b:b + 1].copy()
        ob = O.prefill_kv(one, q[b:b + 1].copy(), k[b:b + 1].copy(), v[b:b + 1].copy(), int(hist[b]), kb, vb, lib)
        assert (ob[0] == out[b]).all() and (kb[0] == kc[b]).all() and (vb[0] == vc[b]).all(), b


def pin_rejects_bad_arguments(lib):
    shape = Shape("pine", 1, 4, 2, 64, 16, 1.0e4)
    q, k, v = w.tokens(shape, "bad", 4)
    kc, vc = w.cache(shape, "bad", 0)
    for call in (lambda: O.prefill_kv(shape, q, k, v, 13, kc, vc, lib),
                 lambda: O.decode(shape, q[:, :1].copy(), k[:, :1].copy(), v[:, :1].copy(),
                                  np.array([16], np.int32), kc, vc, lib),
                 lambda: O.prefill(Shape("pinf", 1, 3, 2, 64, 16, 1.0e4), q[:, :, :3].copy(), k, v, kc, vc, lib)):
        try:
            call()
        except O.OracleError:
            continue
        raise AssertionError("an invalid argument was accepted")


ALL_PINS = [pin_table_closed_forms, pin_rope_complex, pin_rope_identity_norm_relative,
            pin_attention_matches_sdpa, pin_single_key, pin_zero_query, pin_two_key_logistic,
            pin_causality, pin_stage_chain, pin_in_place, pin_decode_mixed_lengths,
            pin_rejects_bad_arguments]
