"""The oracles reproduce their committed tiny-workload fixtures (drift guard)."""
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


def test_w4_oracle_matches_committed_fixture():
    with open(os.path.join(os.path.dirname(G.__file__), "w4_tiny.json")) as f:
        doc = json.load(f)
    res = G.w4_tiny()
    for name, meta in doc["arrays"].items():
        assert list(res[name].shape) == meta["shape"], name
        assert G.digest(res[name]) == meta["sha256"], name
