"""Writes tests/golden/tiny_chain.json from the CPU oracle alone.

The paper prints no numerical worked example for attention, so this fixture holds
the oracle's own result on the tiny workload (4 query heads, 2 KV heads,
head_dim 64, theta 1e4, static max 32): prefill over 16 tokens, prefill_kv of 8
tokens over those 16, then 4 decodes (Section 4.1, scenario 2).  It guards the
oracle against unnoticed drift; the oracle itself is pinned by
tests/oracle_pins.py.  Run:  python tests/golden/make_golden.py
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


def digest(a):
    return hashlib.sha256(np.ascontiguousarray(a, np.uint16).tobytes()).hexdigest()


def main():
    res = tiny_chain()
    doc = {"source": "oracle/attn_oracle.c on the tiny workload (synthetic/workloads.py TINY, tag 'chain', seed 0)",
           "arrays": {name: {"shape": list(a.shape), "sha256": digest(a),
                             "first8_bf16_hex": [f"{int(x):04x}" for x in a.reshape(-1)[:8]]}
                      for name, a in res.items()}}
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "tiny_chain.json"), "w") as f:
        json.dump(doc, f, indent=1)
        f.write("\n")


if __name__ == "__main__":
    main()
