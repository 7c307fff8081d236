"""Pins of the fp64 attention oracle against what the mathematics fixes.

The paper (Sec. 3.1) states only that the target scores the K candidates in
one forward pass against its cache; the oracle writes out softmax attention
with causal masking inside the draft block.  These tests tie it to closed
forms, library routines and the paper's own degenerate case (K = 1 is ordinary
autoregressive decoding, ablation on the draft length K), so that a dropped
scale, a sign, an off-by-one in the causal window, a wrong GQA mapping or a
wrong page/slot index fails at least one of them.
"""
import math

import numpy as np
import pytest
from scipy.special import logsumexp, softmax

from paper_2505_12728_gb300.workloads import (bf16_bits_to_f32, f32_to_bf16_bits,
                                              make_attention_case)

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


def _layer(case):
    return case.q[0], case.k_cache[0], case.v_cache[0], case.block_table[0], case.seq_lens


def _gather_tokens(cache_bits, block_table_row, T, h_kv, page_size=16):
    """Contiguous [T][d] float64 copy of one head's cached tokens (test-side
    indexing, independent of the oracle's)."""
    t = np.arange(T)
    pages = block_table_row[t // page_size]
    return bf16_bits_to_f32(cache_bits[pages, h_kv, t % page_size, :]).astype(np.float64)


def test_single_visible_key_returns_its_value(oracle_mod):
    # n_q = 1 with an empty prefix: one visible key, o = v_0, lse = s_0.
    case = make_attention_case(B=2, n_q=1, H_q=4, H_kv=2, d=64, prefix_lens=[0, 0], seed=11)
    q, kc, vc, bt, sl = _layer(case)
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=2)
    for b in range(2):
        for h in range(4):
            kv = h // 2
            k0 = _gather_tokens(kc, bt[b], 1, kv)[0]
            v0 = _gather_tokens(vc, bt[b], 1, kv)[0]
            qv = bf16_bits_to_f32(q[b, 0, h]).astype(np.float64)
            np.testing.assert_allclose(out[b, 0, h], v0, rtol=0, atol=1e-15)
            assert lse[b, 0, h] == pytest.approx(float(qv @ k0) / math.sqrt(64), abs=1e-12)


@pytest.mark.parametrize("prefix", [0, 1, 15, 16, 17, 31, 32, 33, 100])
def test_zero_query_averages_the_causal_window(oracle_mod, prefix):
    # q = 0 makes every visible score 0: o = mean of the visible values and
    # lse = ln(count).  Row i sees prefix + i + 1 keys (causal draft block).
    n_q = 5
    case = make_attention_case(B=1, n_q=n_q, H_q=2, H_kv=1, d=64, prefix_lens=[prefix], seed=3)
    q, kc, vc, bt, sl = _layer(case)
    q = np.zeros_like(q)
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=1)
    vals = _gather_tokens(vc, bt[0], prefix + n_q, 0)
    for i in range(n_q):
        count = prefix + i + 1
        for h in range(2):
            np.testing.assert_allclose(out[0, i, h], vals[:count].mean(axis=0), rtol=0, atol=1e-12)
            assert lse[0, i, h] == pytest.approx(math.log(count), abs=1e-12)


def test_two_keys_follow_the_logistic_weight(oracle_mod):
    # Two visible keys with scores s0 = scale*a and s1 = 0: the weight of key 0
    # is the logistic function 1/(1+exp(-s0)), lse = log(1 + exp(s0)).
    d = 64
    case = make_attention_case(B=1, n_q=1, H_q=1, H_kv=1, d=d, prefix_lens=[1], seed=5)
    q, kc, vc, bt, sl = _layer(case)
    a = 3.0
    q = np.zeros_like(q)
    q[0, 0, 0, 0] = f32_to_bf16_bits(np.array([a], np.float32))[0]
    kc = kc.copy()
    p0, s0 = bt[0, 0], 0
    kc[p0, 0, 0, :] = 0
    kc[p0, 0, 0, 0] = f32_to_bf16_bits(np.array([1.0], np.float32))[0]   # <q,k0> = a
    kc[p0, 0, 1, :] = 0                                                    # <q,k1> = 0
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=1)
    s = a / math.sqrt(d)
    w0 = 1.0 / (1.0 + math.exp(-s))
    v = _gather_tokens(vc, bt[0], 2, 0)
    np.testing.assert_allclose(out[0, 0, 0], w0 * v[0] + (1 - w0) * v[1], rtol=0, atol=1e-12)
    assert lse[0, 0, 0] == pytest.approx(float(np.logaddexp(s, 0.0)), abs=1e-12)


@pytest.mark.parametrize("H_q,H_kv", [(8, 1), (8, 2), (28, 4), (7, 7)])
def test_gqa_maps_query_heads_to_contiguous_kv_groups(oracle_mod, H_q, H_kv):
    # Constant values per KV head: query head h must read KV head h // (H_q/H_kv).
    case = make_attention_case(B=1, n_q=2, H_q=H_q, H_kv=H_kv, d=64, prefix_lens=[40], seed=7)
    q, kc, vc, bt, sl = _layer(case)
    vc = vc.copy()
    consts = np.arange(1, H_kv + 1, dtype=np.float32)
    for kv in range(H_kv):
        vc[:, kv] = f32_to_bf16_bits(np.full(vc[:, kv].shape, consts[kv], np.float32))
    out, _ = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=H_kv)
    g = H_q // H_kv
    for h in range(H_q):
        np.testing.assert_allclose(out[0, :, h], consts[h // g], rtol=0, atol=1e-12)


def test_page_table_and_slot_indexing(oracle_mod):
    # Values equal the logical token position (exact in bf16 up to 256); with
    # q = 0 row i returns the mean position (prefix + i) / 2.  Pages are a
    # random permutation of a pool with unused spare pages.
    n_q, prefixes = 4, [0, 37, 200]
    case = make_attention_case(B=3, n_q=n_q, H_q=2, H_kv=2, d=64, prefix_lens=prefixes, seed=9,
                               spare_pages=5)
    q, kc, vc, bt, sl = _layer(case)
    q = np.zeros_like(q)
    vc = np.zeros_like(vc)
    for b in range(3):
        for t in range(int(sl[b])):
            vc[bt[b, t // 16], :, t % 16, :] = f32_to_bf16_bits(np.array([t], np.float32))[0]
    out, _ = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=2)
    for b, L in enumerate(prefixes):
        for i in range(n_q):
            np.testing.assert_allclose(out[b, i], (L + i) / 2.0, rtol=0, atol=1e-12)


def test_verify_rows_equal_sequential_decodes(oracle_mod):
    # A k-row verification equals k sequential decodes: row i is one decode
    # step at position L+i over the first L+i+1 cached tokens (the K = 1
    # degenerate case of the draft-length ablation).
    n_q, H_q, H_kv, d = 6, 8, 2, 128
    case = make_attention_case(B=2, n_q=n_q, H_q=H_q, H_kv=H_kv, d=d, prefix_lens=[50, 129],
                               seed=13)
    q, kc, vc, bt, sl = _layer(case)
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=H_kv)
    scale = 1.0 / math.sqrt(d)
    for b in range(2):
        L = int(sl[b]) - n_q
        for i in range(n_q):
            for h in range(H_q):
                K = _gather_tokens(kc, bt[b], L + i + 1, h // (H_q // H_kv))
                Vv = _gather_tokens(vc, bt[b], L + i + 1, h // (H_q // H_kv))
                qv = bf16_bits_to_f32(q[b, i, h]).astype(np.float64)
                o, l = oracle_mod.decode_attention(qv, K, Vv, scale)
                np.testing.assert_allclose(out[b, i, h], o, rtol=0, atol=1e-12)
                assert lse[b, i, h] == pytest.approx(l, abs=1e-12)


def test_single_row_verify_of_truncated_sequence_matches_row_i(oracle_mod):
    # Verifying only draft row i against the sequence cut at L+i+1 tokens
    # gives the same row as the full k-row verification.
    n_q, H_q, H_kv, d = 5, 4, 4, 64
    case = make_attention_case(B=1, n_q=n_q, H_q=H_q, H_kv=H_kv, d=d, prefix_lens=[70], seed=17)
    q, kc, vc, bt, sl = _layer(case)
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=H_kv)
    for i in range(n_q):
        sl_i = np.array([int(sl[0]) - n_q + i + 1], np.int32)
        o1, l1 = oracle_mod.verify_attention(q[:, i:i + 1], kc, vc, bt, sl_i, H_kv=H_kv)
        np.testing.assert_allclose(o1[0, 0], out[0, i], rtol=0, atol=1e-12)
        np.testing.assert_allclose(l1[0, 0], lse[0, i], rtol=0, atol=1e-12)


def test_matches_scipy_softmax_and_logsumexp(oracle_mod):
    # Library routines: lse = scipy logsumexp of the scaled scores, o =
    # scipy softmax(scores) @ V, for every row, with an explicit scale.
    n_q, H_q, H_kv, d = 3, 6, 3, 64
    case = make_attention_case(B=2, n_q=n_q, H_q=H_q, H_kv=H_kv, d=d, prefix_lens=[33, 64],
                               seed=19)
    q, kc, vc, bt, sl = _layer(case)
    scale = 0.3
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=H_kv, scale=scale)
    g = H_q // H_kv
    for b in range(2):
        T = int(sl[b])
        for h in range(H_q):
            K = _gather_tokens(kc, bt[b], T, h // g)
            Vv = _gather_tokens(vc, bt[b], T, h // g)
            Q = bf16_bits_to_f32(q[b, :, h]).astype(np.float64)
            S = scale * (Q @ K.T)
            for i in range(n_q):
                vis = T - n_q + i + 1
                assert lse[b, i, h] == pytest.approx(float(logsumexp(S[i, :vis])), abs=1e-12)
                np.testing.assert_allclose(out[b, i, h], softmax(S[i, :vis]) @ Vv[:vis],
                                           rtol=0, atol=1e-12)


def test_default_scale_is_inverse_sqrt_head_dim(oracle_mod):
    case = make_attention_case(B=1, n_q=2, H_q=2, H_kv=1, d=128, prefix_lens=[20], seed=23)
    q, kc, vc, bt, sl = _layer(case)
    o0, l0 = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=1, scale=0.0)
    o1, l1 = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=1, scale=1 / math.sqrt(128))
    np.testing.assert_array_equal(o0, o1)
    np.testing.assert_array_equal(l0, l1)


def test_physical_page_order_does_not_matter(oracle_mod):
    case = make_attention_case(B=2, n_q=3, H_q=4, H_kv=2, d=64, prefix_lens=[45, 90], seed=29,
                               spare_pages=3)
    q, kc, vc, bt, sl = _layer(case)
    out, lse = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=2)
    rng = np.random.default_rng(1)
    perm = rng.permutation(kc.shape[0])          # new physical slot of old page p is perm[p]
    kc2 = np.empty_like(kc)
    vc2 = np.empty_like(vc)
    kc2[perm] = kc
    vc2[perm] = vc
    bt2 = np.where(bt >= 0, perm[np.maximum(bt, 0)], -1).astype(np.int32)
    out2, lse2 = oracle_mod.verify_attention(q, kc2, vc2, bt2, sl, H_kv=2)
    np.testing.assert_array_equal(out, out2)
    np.testing.assert_array_equal(lse, lse2)


def test_row_selection_computes_only_selected_rows(oracle_mod):
    case = make_attention_case(B=2, n_q=3, H_q=4, H_kv=2, d=64, prefix_lens=[10, 20], seed=31)
    q, kc, vc, bt, sl = _layer(case)
    full, lfull = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=2)
    sel, lsel = oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=2, select=(1, 2, 3))
    np.testing.assert_array_equal(sel[1, 2, 3], full[1, 2, 3])
    assert lsel[1, 2, 3] == lfull[1, 2, 3]
    assert np.isnan(sel[0]).all() and np.isnan(lsel[0]).all()


def test_out_of_range_page_is_an_error(oracle_mod):
    case = make_attention_case(B=1, n_q=2, H_q=2, H_kv=1, d=64, prefix_lens=[30], seed=37)
    q, kc, vc, bt, sl = _layer(case)
    bt = bt.copy()
    bt[0, 1] = kc.shape[0] + 3
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.verify_attention(q, kc, vc, bt, sl, H_kv=1)
