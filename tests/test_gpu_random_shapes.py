"""Seeded random-shape parity sweep of both calls against the oracle (GPU).

Shapes, prefix lengths (with tile- and page-boundary values mixed in), split
counts, vocabulary sizes (both acceptance paths, aligned or not), modes and
temperatures are drawn from one seeded generator, so that paths the fixed
grids of the other tests miss still meet the oracle.  Tolerances are those
of the other parity tests.
"""
import numpy as np
import pytest

from paper_2505_12728_gb300.workloads import make_accept_case, make_attention_case
from tests.gpu_helpers import (assert_attention_close, compare_accept, oracle_accept,
                               oracle_attention, require_gpu, run_accept, run_attention)

pytestmark = pytest.mark.gpu

BOUNDARY_PREFIXES = [0, 1, 15, 16, 17, 63, 64, 65, 127, 128, 129, 511, 512, 513]
VOCABS = [2, 3, 5, 100, 1001, 4096, 32000, 32768, 32769, 40000, 65536, 65537, 131072, 152064,
          160000, 200003]


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def test_random_attention_shapes_match_oracle(oracle_mod):
    rng = np.random.default_rng(20261202)
    for c in range(80):
        d = int(rng.choice([64, 128]))
        H_kv = int(rng.integers(1, 9))
        H_q = H_kv * int(rng.choice([1, 2, 4, 7, 8]))
        n_q = int(rng.integers(1, 17))
        B = int(rng.integers(1, 25))
        prefixes = [int(rng.choice(BOUNDARY_PREFIXES)) if rng.random() < 0.3
                    else int(rng.integers(0, 5000)) for _ in range(B)]
        # keep the oracle's work per case to ~1e10 flops
        while B > 1 and n_q * H_q * sum(p + n_q for p in prefixes) * d * 2 > 1e10:
            B -= 1
            prefixes = prefixes[:B]
        splits = int(rng.choice([0, 0, 0, 1, 2, 3, 7, 37, 200]))
        case = make_attention_case(B, n_q, H_q, H_kv, d, prefixes, seed=300000 + c,
                                   spare_pages=int(rng.integers(0, 4)))
        out, lse = run_attention(case, num_splits=splits)
        ref_out, ref_lse = oracle_attention(oracle_mod, case)
        try:
            assert_attention_close(out, lse, ref_out, ref_lse)
        except AssertionError as e:
            raise AssertionError(f"case {c}: B={B} n_q={n_q} H_q={H_q} H_kv={H_kv} d={d} "
                                 f"splits={splits} prefixes={prefixes}: {e}") from None


def test_random_acceptance_shapes_match_oracle(oracle_mod):
    rng = np.random.default_rng(20261203)
    excluded = 0
    sequences = 0
    for c in range(60):
        V = int(rng.choice(VOCABS))
        k = int(rng.integers(1, 17))
        B = int(rng.integers(1, 33)) if V < 100000 else int(rng.integers(1, 12))
        mode = str(rng.choice(["sampling", "greedy", "alternate"]))
        inp = make_accept_case(B, k, V, seed=400000 + c, mode=mode,
                               logit_std=float(rng.choice([1.0, 3.0, 6.0])))
        if mode != "greedy" and rng.random() < 0.3:
            inp.temperature = np.where(inp.temperature > 0, rng.choice([0.5, 0.8, 1.3]),
                                       0.0).astype(np.float32)
        n, toks, ratio = run_accept(inp)
        ref = oracle_accept(oracle_mod, inp)
        try:
            excluded += compare_accept(ref, n, toks, ratio)  # bit-exact outside the margin
        except AssertionError as e:
            raise AssertionError(f"case {c}: B={B} k={k} V={V} mode={mode}: {e}") from None
        sequences += B
    # draws within 1e-6 of a CDF boundary are frequent only for very flat
    # targets over large vocabularies; over the sweep they stay rare
    assert excluded <= 0.05 * sequences, (excluded, sequences)
