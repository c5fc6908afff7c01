"""The oracle reproduces its committed tiny-workload fixture (drift guard)."""
import json
import os

from tests.golden import make_golden as G


def test_oracle_matches_committed_fixture():
    with open(os.path.join(os.path.dirname(G.__file__), "tiny_chain.json")) as f:
        doc = json.load(f)
    res = G.tiny_chain()
    for name, meta in doc["arrays"].items():
        assert list(res[name].shape) == meta["shape"], name
        assert G.digest(res[name]) == meta["sha256"], name
