"""Writes tests/golden/tiny_chain.json and tests/golden/w4_tiny.json from the CPU oracles alone.

The paper prints no numerical worked example for attention, so this fixture holds
the oracle's own result on the tiny workload (4 query heads, 2 KV heads,
head_dim 64, theta 1e4, static max 32): prefill over 16 tokens, prefill_kv of 8
tokens over those 16, then 4 decodes (Section 4.1, scenario 2).  It guards the
oracle against unnoticed drift; the oracle itself is pinned by
tests/oracle_pins.py.  w4_tiny.json does the same for the W4BF16 oracle
(oracle/w4_oracle.py, pinned by tests/w4_oracle_pins.py): the tile stream of a small
matrix, its GEMV, RMSNorm, the prefill-side GEMM, one decode step and one prefill_kv chunk
of the block around attention, every float64 result rounded to bf16 before it is hashed.
Run:  python tests/golden/make_golden.py
"""
import hashlib
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import oracle as O  # noqa: E402
from synthetic import workloads as w  # noqa: E402


def tiny_chain():
    s = w.TINY
    q, k, v = w.tokens(s, "chain", 28)
    kc, vc = w.cache(s, "chain", 0)
    out = {"prefill": O.prefill(s, q[:, :16].copy(), k[:, :16].copy(), v[:, :16].copy(), kc, vc),
           "prefill_kv": O.prefill_kv(s, q[:, 16:24].copy(), k[:, 16:24].copy(), v[:, 16:24].copy(), 16, kc, vc)}
    for t in range(24, 28):
        out[f"decode{t}"] = O.decode(s, q[:, t:t + 1].copy(), k[:, t:t + 1].copy(), v[:, t:t + 1].copy(),
                                     np.full(s.batch, t, np.int32), kc, vc)
    out["k_cache"], out["v_cache"] = kc, vc
    return out


def w4_tiny():
    from oracle import w4_oracle as W
    from synthetic import gen
    from synthetic.workloads import Shape
    N, K, M = 40, 256, 3
    codes = gen.uint4_codes("golden_w4", "codes", (N, K))
    zeros = gen.uint4_codes("golden_w4", "zeros", (N, K // 128))
    scales = gen.normal_bf16("golden_w4", "scales", (N, K // 128), 0.02)
    x = gen.normal_bf16("golden_w4", "x", (M, K), 1.0)
    gamma = gen.normal_bf16("golden_w4", "gamma", (K,), 0.5)
    out = {"tiles": W.write_tiles(codes, scales, zeros).view(np.uint16),
           "gemv": W.to_bf16_bits(W.gemv(codes, scales, zeros, x)),
           "rmsnorm": W.rmsnorm(x, gamma, 1e-6),
           "gemm": W.to_bf16_bits(W.gemm_bf16w(codes, scales, zeros, x))}
    sh = Shape("golden_w4_block", 2, 4, 2, 64, 64, 1.0e4)
    qd, kd, hidden = 256, 128, 256
    wq = (gen.uint4_codes("golden_w4", "qkv_c", (qd + 2 * kd, hidden)),
          gen.normal_bf16("golden_w4", "qkv_s", (qd + 2 * kd, hidden // 128), 0.02),
          gen.uint4_codes("golden_w4", "qkv_z", (qd + 2 * kd, hidden // 128)))
    wo = (gen.uint4_codes("golden_w4", "o_c", (hidden, qd)),
          gen.normal_bf16("golden_w4", "o_s", (hidden, qd // 128), 0.02),
          gen.uint4_codes("golden_w4", "o_z", (hidden, qd // 128)))
    xb = gen.normal_bf16("golden_w4", "xb", (2, hidden), 1.0)
    gb = gen.normal_bf16("golden_w4", "gb", (hidden,), 0.5)
    kc, vc = w.cache(sh, "golden_w4", 20, fill="random")
    out["block_h"] = W.decode_layer(sh, xb, gb, 1e-6, wq, wo, np.array([5, 20], np.int32), kc, vc)
    out["block_k_cache"], out["block_v_cache"] = kc, vc
    # the prefill side: a 7-token chunk of each of the two sequences over 21 history tokens
    xp = gen.normal_bf16("golden_w4", "xp", (2, 7, hidden), 1.0)
    kc, vc = w.cache(sh, "golden_w4_prefill", 21, fill="random")
    out["prefill_block_h"] = W.prefill_layer(sh, xp, gb, 1e-6, wq, wo, 21, kc, vc)
    out["prefill_block_k_cache"], out["prefill_block_v_cache"] = kc, vc
    return out


def digest(a):
    return hashlib.sha256(np.ascontiguousarray(a, np.uint16).tobytes()).hexdigest()


def write(name, source, res):
    doc = {"source": source,
           "arrays": {key: {"shape": list(a.shape), "sha256": digest(a),
                            "first8_bf16_hex": [f"{int(x):04x}" for x in a.reshape(-1)[:8]]}
                      for key, a in res.items()}}
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), name), "w") as f:
        json.dump(doc, f, indent=1)
        f.write("\n")


def main():
    write("tiny_chain.json", "oracle/attn_oracle.c on the tiny workload (synthetic/workloads.py TINY, tag 'chain', "
          "seed 0)", tiny_chain())
    write("w4_tiny.json", "oracle/w4_oracle.py (with oracle/attn_oracle.c for the block's attention) on stream "
          "'golden_w4', seed 0", w4_tiny())


if __name__ == "__main__":
    main()
