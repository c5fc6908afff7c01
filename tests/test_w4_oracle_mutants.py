"""The W4BF16 oracle's pins are strong enough: every planted mistake in a copy of the
oracle fails one of them.

Each mutant is oracle/w4_oracle.py with one plausible mistake substituted in (a wrong
nibble order or tile transpose, a tile writer that misplaces a scale byte, a code row or a
zero point, a dropped zero point, a wrong group, a wrong bf16 decode
or rounding, RMSNorm without eps or gamma or with a sum for the mean, a block without its
residual or RMSNorm, k and v swapped, q read from the wrong rows, GEMM weights not rounded; the
prefill block without its residual or RMSNorm, with k and v swapped, q from the wrong rows,
unrounded projection weights, or its history ignored),
loaded as a separate module.  The real oracle is never modified.
"""
import os
import types

import pytest

from oracle import w4_oracle as W
from tests import w4_oracle_pins as P

MUTANTS = {
    "nibbles_in_order": ("NIBBLE_SHIFT = (0, 16, 4, 20, 8, 24, 12, 28)", "NIBBLE_SHIFT = (0, 4, 8, 12, 16, 20, 24, 28)"),
    "tile_words_not_transposed": ("words = words.transpose(0, 2, 1, 3)", "words = words.transpose(0, 1, 2, 3)"),
    "zero_points_not_transposed": ("zeros = zeros.transpose(0, 2, 1)", "zeros = zeros.transpose(0, 1, 2)"),
    "zero_point_ignored": ("return (q - z) * s", "return q * s"),
    "scales_of_the_wrong_group": ("s = np.repeat(bf16_to_f64(scales_bf16), GROUP, axis=-1)",
                                  "s = np.repeat(bf16_to_f64(scales_bf16)[..., ::-1], GROUP, axis=-1)"),
    "bf16_decode_shift": ("<< np.uint32(16)).view(np.float32)", "<< np.uint32(15)).view(np.float32)"),
    "rounding_truncates": ("np.rint(np.ldexp(m, 8))", "np.trunc(np.ldexp(m, 8))"),
    "rmsnorm_without_eps": ("np.mean(x * x, axis=-1, keepdims=True) + eps)", "np.mean(x * x, axis=-1, keepdims=True))"),
    "rmsnorm_without_gamma": ("return to_bf16_bits(x * r * bf16_to_f64(gamma_bf16))", "return to_bf16_bits(x * r)"),
    "rmsnorm_sum_for_mean": ("np.mean(x * x, axis=-1", "np.sum(x * x, axis=-1"),
    "block_without_residual": ("return to_bf16_bits(bf16_to_f64(x_bf16) + gemv(*wo, o))", "return to_bf16_bits(gemv(*wo, o))"),
    "block_without_rmsnorm": ("xn = rmsnorm(x_bf16, gamma_bf16, eps)", "xn = x_bf16"),
    "block_k_v_swapped": ("v = qkv[:, qd + kd:].reshape(B, 1,", "v = qkv[:, qd:qd + kd].reshape(B, 1,"),
    "block_q_from_wrong_rows": ("q = qkv[:, :qd].reshape(B, 1,", "q = qkv[:, kd:kd + qd].reshape(B, 1,"),
    "writer_scale_bytes_swapped": ("buf[at.ravel()] = (s & 0xFF)", "buf[at.ravel()] = (s >> 8)"),
    "writer_code_byte_ignores_row": ("+ 64 * (n % TILE_ROWS) + 4 *", "+ 4 *"),
    "writer_zero_point_in_scale_bytes": ("buf[(rec * TILE_BYTES + ZERO_OFFSET + n % TILE_ROWS)",
                                         "buf[(rec * TILE_BYTES + SCALE_OFFSET + n % TILE_ROWS)"),
    "prefill_block_without_residual": ("return to_bf16_bits(bf16_to_f64(x2) + gemm_bf16w(*wo, o)).reshape(B, S, hidden)",
                                       "return to_bf16_bits(gemm_bf16w(*wo, o)).reshape(B, S, hidden)"),
    "prefill_block_without_rmsnorm": ("xn = rmsnorm(x2, gamma_bf16, eps)", "xn = x2"),
    "prefill_block_k_v_swapped": ("v = qkv[:, qd + kd:].reshape(B, S", "v = qkv[:, qd:qd + kd].reshape(B, S"),
    "prefill_block_q_from_wrong_rows": ("q = qkv[:, :qd].reshape(B, S", "q = qkv[:, kd:kd + qd].reshape(B, S"),
    "prefill_block_weights_not_rounded": ("qkv = to_bf16_bits(gemm_bf16w(*wqkv, xn))", "qkv = to_bf16_bits(gemv(*wqkv, xn))"),
    "prefill_block_history_ignored": ("o = attn_oracle.prefill_kv(shape, q, k, v, int(hist), k_cache, v_cache)",
                                      "o = attn_oracle.prefill_kv(shape, q, k, v, 0, k_cache, v_cache)"),
    "gemm_weights_not_rounded": ("@ bf16_to_f64(dequant_bf16(codes, scales_bf16, zeros)).T",
                                 "@ dequant(codes, scales_bf16, zeros).T"),
}


@pytest.fixture(scope="module")
def source():
    with open(os.path.join(os.path.dirname(W.__file__), "w4_oracle.py")) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, source):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name} not unique in the oracle source"
    mod = types.ModuleType(f"w4_oracle_{name}")
    exec(compile(source.replace(old, new), f"<mutant {name}>", "exec"), mod.__dict__)
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(mod)
        except (AssertionError, ValueError, IndexError, FloatingPointError):
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake {name}"
