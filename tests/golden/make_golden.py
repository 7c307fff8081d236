"""Write the oracle regression fixtures in this folder.

The paper prints no worked numeric example of the verification step, so no
stored value here comes from the paper.  These fixtures are written by this
script, which calls only the CPU oracle (``oracle/``) on seeded synthetic
inputs; they guard the oracle against unnoticed changes.  A change to a stored
value must name, in its commit message, the passage of the paper (or the
reading of it) that justifies it.

Run from the repository root:  python tests/golden/make_golden.py
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

from oracle import oracle  # noqa: E402
from paper_2505_12728_gb300.workloads import make_accept_case, make_attention_case  # noqa: E402

ATTN_CASE = dict(B=2, n_q=4, H_q=8, H_kv=2, d=64, prefix_lens=[40, 77], seed=2024)
ACCEPT_CASE = dict(B=24, k=4, V=64, seed=2025, mode="alternate")


def attention_fixture():
    c = make_attention_case(**ATTN_CASE)
    out, lse = oracle.verify_attention(c.q[0], c.k_cache[0], c.v_cache[0], c.block_table[0],
                                       c.seq_lens, H_kv=ATTN_CASE["H_kv"])
    return dict(case=ATTN_CASE, lse=[round(float(x), 12) for x in lse.ravel()],
                out_row_sums=[round(float(x), 12) for x in out.sum(axis=-1).ravel()],
                out_first=[round(float(x), 12) for x in out[..., 0].ravel()])


def accept_fixture():
    a = make_accept_case(**ACCEPT_CASE)
    r = oracle.accept(a.target_logits, a.draft_probs, a.draft_tokens, a.uniforms, a.temperature)
    return dict(case=ACCEPT_CASE, num_accepted=r["num_accepted"].tolist(),
                out_tokens=r["out_tokens"].tolist(),
                accept_ratio=[round(float(x), 12) for x in r["accept_ratio"].ravel()])


if __name__ == "__main__":
    with open(os.path.join(HERE, "oracle_attention_small.json"), "w") as f:
        json.dump(attention_fixture(), f, indent=1)
    with open(os.path.join(HERE, "oracle_accept_small.json"), "w") as f:
        json.dump(accept_fixture(), f, indent=1)
