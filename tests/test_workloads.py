"""The seeded input generators shared by the oracle tests, the GPU parity tests
and the benchmark: the structure they promise (paged layout, sequence
lengths, the named workloads' shapes, the draft distributions and tokens,
the exact-integer draft-tail inputs) and their determinism."""
import numpy as np
import pytest

from paper_2505_12728_gb300.workloads import (HIDDEN_SIZES, WORKLOADS, bf16_bits_to_f32,
                                              f32_to_bf16_bits, make_accept_case,
                                              make_accept_inputs, make_attention_case,
                                              make_compress_case, make_draft_tail_case,
                                              prefix_lengths, temperatures)


def test_bf16_rounding_is_round_to_nearest_even():
    x = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -9, -2.5, 0.0, np.inf], np.float32)
    got = bf16_bits_to_f32(f32_to_bf16_bits(x))
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties to the even mantissa (1)
    np.testing.assert_array_equal(got, np.array([1.0, 1.0, 1.0 + 2.0 ** -7, -2.5, 0.0, np.inf],
                                                np.float32))


@pytest.mark.parametrize("prefixes,n_q,max_pages", [([0, 15, 16, 200], 4, None),
                                                    ([37], 5, 40), ([1000, 1], 8, None)])
def test_paged_cache_layout(prefixes, n_q, max_pages):
    case = make_attention_case(len(prefixes), n_q, 8, 2, 64, prefixes, seed=3, layers=2,
                               spare_pages=5, max_pages=max_pages)
    B = len(prefixes)
    np.testing.assert_array_equal(case.seq_lens, np.array(prefixes) + n_q)
    pages = (case.seq_lens + 15) // 16
    assert case.k_cache.shape[1] == int(pages.sum()) + 5          # the pool, with spare pages
    for l in range(2):
        used = []
        for b in range(B):
            row = case.block_table[l, b]
            assert (row[:pages[b]] >= 0).all() and (row[pages[b]:] == -1).all()
            used.extend(row[:pages[b]].tolist())
        # distinct physical pages inside the pool; the spare pages are never referenced
        assert len(set(used)) == len(used) == int(pages.sum())
        assert max(used) < case.k_cache.shape[1]
    if max_pages is not None:
        assert case.block_table.shape[2] == max_pages


def test_attention_case_is_deterministic_and_seed_dependent():
    a = make_attention_case(2, 4, 8, 8, 64, [50, 70], seed=11)
    b = make_attention_case(2, 4, 8, 8, 64, [50, 70], seed=11)
    c = make_attention_case(2, 4, 8, 8, 64, [50, 70], seed=12)
    for x, y in ((a.q, b.q), (a.k_cache, b.k_cache), (a.block_table, b.block_table)):
        np.testing.assert_array_equal(x, y)
    assert not np.array_equal(a.q, c.q)


@pytest.mark.parametrize("name,lo,hi", [("tiny", 640, 640), ("image7b", 3008, 3008),
                                        ("gqa", 1200, 3600), ("video", 4864, 4864),
                                        ("long", 8192, 32768)])
def test_named_workload_prefixes(name, lo, hi):
    wl = WORKLOADS[name]
    L = prefix_lengths(wl, np.random.default_rng([wl.seed, 0xA77]))
    assert L.shape == (wl.B,) and (L >= lo).all() and (L <= hi).all()
    assert wl.H_q % wl.H_kv == 0 and wl.d in (64, 128)
    assert wl.V in HIDDEN_SIZES


def test_named_workload_visual_token_counts():
    # 5 LLaVA images of 576 tokens + 128 text tokens; 32 video frames of 144
    # tokens + 256 text tokens (the prefix lengths quoted in the descriptions)
    assert WORKLOADS["image7b"].prefix == ("fixed", 5 * 576 + 128)
    assert WORKLOADS["video"].prefix == ("fixed", 32 * 144 + 256)
    assert WORKLOADS["tiny"].prefix == ("fixed", 576 + 64)


@pytest.mark.parametrize("mode", ["sampling", "greedy", "alternate"])
def test_accept_case_draft_distributions_and_tokens(mode):
    inp = make_accept_case(6, 3, 50, seed=[5, 7], mode=mode)
    B, k, V = inp.shape
    assert (B, k, V) == (6, 3, 50)
    np.testing.assert_array_equal(inp.temperature, temperatures(mode, B))
    np.testing.assert_allclose(inp.draft_probs.sum(axis=-1, dtype=np.float64), 1.0, atol=1e-5)
    assert (inp.draft_probs >= 0).all()
    assert ((inp.draft_tokens >= 0) & (inp.draft_tokens < V)).all()
    assert ((inp.uniforms >= 0) & (inp.uniforms < 1)).all()
    for b in range(B):
        for i in range(k):
            x = inp.draft_tokens[b, i]
            if inp.temperature[b] > 0:
                assert inp.draft_probs[b, i, x] > 0        # drawn from q_i
            else:
                assert x == int(np.argmax(inp.draft_probs[b, i]))


def test_accept_draft_tokens_follow_q():
    # sampling drafts are categorical draws from q: on one row repeated many
    # times the empirical frequencies approach q
    inp = make_accept_case(4000, 1, 4, seed=9, draft_sharpness=0.3, logit_std=1.0)
    q = inp.draft_probs[:, 0, :].astype(np.float64)
    hits = np.zeros(4)
    for b in range(4000):
        hits[inp.draft_tokens[b, 0]] += 1.0
    expected = q.sum(axis=0)
    assert np.abs(hits - expected).max() < 5 * np.sqrt(expected.max())


def test_named_workload_accept_inputs_shapes():
    for name, wl in WORKLOADS.items():
        if wl.V > 32000:
            continue  # the 152064-token workloads are checked on the GPU side
        inp = make_accept_inputs(wl)
        assert inp.shape == (wl.B, wl.k, wl.V)


def test_exact_draft_tail_inputs_are_small_integers():
    case = make_draft_tail_case(4, 64, 100, seed=2, exact=True)
    h = bf16_bits_to_f32(case.hidden)
    w = bf16_bits_to_f32(case.weight)
    assert set(np.unique(h).tolist()) <= set(range(-3, 4))
    scale = np.abs(w[w != 0]).min()
    assert np.log2(scale) == np.round(np.log2(scale))               # a power of two
    np.testing.assert_array_equal(np.round(w / scale), w / scale)  # integer multiples of it
    assert np.abs(w / scale).max() <= 3


def test_compress_case_scales():
    queries, features = make_compress_case(3, 200, 16, 512, seed=4, q_std=2.0)
    assert queries.shape == (16, 512) and features.shape == (3, 200, 512)
    f = bf16_bits_to_f32(features).astype(np.float64)
    qv = bf16_bits_to_f32(queries).astype(np.float64)
    assert abs(f.std() - 1.0) < 0.02
    scores = np.einsum("cd,fnd->fcn", qv, f)
    assert abs(scores.std() - 2.0) < 0.1                           # scores ~ N(0, q_std^2)
