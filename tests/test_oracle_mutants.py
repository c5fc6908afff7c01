"""The pins are strong enough: every planted mistake in a copy of the oracle fails one.

Each mutant is the oracle source with one plausible mistake substituted in (a
wrong sign, a dropped term, a wrong index, an off-by-one), built into a temporary
library.  The real oracle is never modified.
"""
import os

import pytest

from oracle import oracle as O
from tests import oracle_pins as P

MUTANTS = {
    "rope_sign": ("y[j] = ac - bs;", "y[j] = ac + bs;"),
    "rope_second_half_sign": ("y[j + half] = bc + as;", "y[j + half] = bc - as;"),
    "rope_frequency": ("-(2.0 * j) / (double)head_dim", "-(1.0 * j) / (double)head_dim"),
    "rope_pairing": ("float b = bf16_to_float(x[j + half]);", "float b = bf16_to_float(x[2 * j + 1 < head_dim ? 2 * j + 1 : j]);"),
    "dropped_scale": ("s *= scale;", "s *= 1.0;"),
    "causal_excludes_self": ("for (int j = 0; j <= p; ++j) {\n        double s", "for (int j = 0; j < p; ++j) {\n        double s"),
    "causal_sees_next": ("for (int j = 0; j <= p; ++j) {\n        double w", "for (int j = 0; j <= p + (p + 1 < L); ++j) {\n        double w"),
    "gqa_modulo": ("int g = h / (c->n_q_heads / c->n_kv_heads);", "int g = h % c->n_kv_heads;"),
    "v_gets_k": ("v_cache[dst + d] = v[src + d];", "v_cache[dst + d] = k[src + d];"),
    "k_not_rotated": ("k_cache[dst + d] = float_to_bf16(y[d]);", "k_cache[dst + d] = k[src + d];"),
    "q_not_rotated": ("for (int d = 0; d < D; ++d) qr[d] = bf16_to_float(float_to_bf16(qr[d]));",
                      "for (int d = 0; d < D; ++d) qr[d] = bf16_to_float(q_row[d]);"),
    "append_wrong_slot": ("int p = hist[b] + i;\n            for (int g = 0; g < Hkv; ++g) {",
                          "int p = i;\n            for (int g = 0; g < Hkv; ++g) {"),
    "softmax_not_normalised": ("(float)(acc[d] / l)", "(float)(acc[d])"),
}


@pytest.fixture(scope="module")
def source():
    with open(os.path.join(os.path.dirname(O.__file__), "attn_oracle.c")) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, source, tmp_path):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name} not unique in the oracle source"
    src = tmp_path / f"{name}.c"
    src.write_text(source.replace(old, new))
    lib = O.load(O.build(force=True, src=str(src), out=str(tmp_path / f"lib{name}.so")))
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(lib)
        except (AssertionError, O.OracleError, FloatingPointError, ValueError):
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake {name}"
