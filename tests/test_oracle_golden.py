"""The oracle reproduces its stored regression fixtures (tests/golden/)."""
import json
import os

import numpy as np

from tests.golden import make_golden

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(HERE, name)) as f:
        return json.load(f)


def test_attention_fixture(oracle_mod):
    want = _load("oracle_attention_small.json")
    got = make_golden.attention_fixture()
    assert got["case"] == want["case"]
    for key in ("lse", "out_row_sums", "out_first"):
        np.testing.assert_allclose(got[key], want[key], rtol=0, atol=1e-10)


def test_accept_fixture(oracle_mod):
    want = _load("oracle_accept_small.json")
    got = make_golden.accept_fixture()
    assert got["case"] == want["case"]
    assert got["num_accepted"] == want["num_accepted"]
    assert got["out_tokens"] == want["out_tokens"]
    np.testing.assert_allclose(got["accept_ratio"], want["accept_ratio"], rtol=0, atol=1e-10)
