"""Pins of the fp64 acceptance oracle against what the mathematics fixes.

The paper applies the token-wise acceptance-rejection rule of speculative
sampling (Sec. 3.1, Sec. 3.3) and relies on its guarantee that accepted tokens
are samples of the target distribution (Sec. 1).  The oracle is pinned by:
library routines (scipy softmax, numpy argmax/searchsorted), hand-worked small
cases, greedy decoding as plain sequential argmax, an exact reconstruction of
the output distribution by bisection over the uniforms (it must equal p), the
closed-form law of the accepted length, and a Monte-Carlo check of the
emitted tokens.  A flipped inequality, a missing clamp, a residual of q - p,
a wrong row or uniform index, or an unnormalised residual fails one of them.
"""
import math

import numpy as np
import pytest
from scipy.special import softmax
from scipy.stats import chisquare

from paper_2505_12728_gb300.workloads import make_accept_case

ONE_MINUS = np.nextafter(np.float32(1.0), np.float32(0.0))


def _single(oracle_mod, logits, q, tokens, u, tau=1.0):
    logits = np.asarray(logits, np.float32)[None]
    q = np.asarray(q, np.float32)[None]
    tokens = np.asarray(tokens, np.int32)[None]
    u = np.asarray(u, np.float32)[None]
    res = oracle_mod.accept(logits, q, tokens, u, np.array([tau], np.float32))
    return {k: v[0] for k, v in res.items()}


@pytest.mark.parametrize("tau", [1.0, 0.7, 2.0])
def test_target_probs_match_scipy_softmax(oracle_mod, tau):
    rng = np.random.default_rng(0)
    logits = (3 * rng.standard_normal(5000)).astype(np.float32)
    p = oracle_mod.target_probs(logits, tau)
    ref = softmax(logits.astype(np.float64) / tau)
    np.testing.assert_allclose(p, ref, rtol=1e-12, atol=0)


def test_argmax_takes_the_first_maximum(oracle_mod):
    assert oracle_mod.argmax(np.array([1, 5, 5, 2], np.float32)) == 1
    assert oracle_mod.argmax(np.array([7, 5, 7], np.float32)) == 0
    rng = np.random.default_rng(1)
    for _ in range(50):
        x = rng.integers(-3, 3, size=17).astype(np.float32)
        assert oracle_mod.argmax(x) == int(np.argmax(x))


def test_hand_worked_three_token_vocabulary(oracle_mod):
    # p = (1/2, 1/3, 1/6) (logits = log p), q = (1/3, 1/2, 1/6).
    p = np.array([1 / 2, 1 / 3, 1 / 6])
    q = np.array([[1 / 3, 1 / 2, 1 / 6]])
    logits = np.log(np.stack([p, p]))
    # Draft token 0: p/q = 3/2 >= 1, accepted for every u; the bonus row is p.
    r = _single(oracle_mod, logits, q, [0], [ONE_MINUS, 0.1])
    assert r["num_accepted"] == 1 and r["out_tokens"][0] == 0
    assert r["out_tokens"][1] == 0                      # 0.1 < 1/2 -> token 0
    r = _single(oracle_mod, logits, q, [0], [0.3, 0.6])
    assert list(r["out_tokens"]) == [0, 1]              # 1/2 <= 0.6 < 5/6 -> token 1
    # Draft token 1: p/q = 2/3.  u = 0.5 accepts; u = 0.9 rejects and the
    # residual max(0, p - q) = (1/6, 0, 0) puts all mass on token 0.
    r = _single(oracle_mod, logits, q, [1], [0.5, 0.99])
    assert r["num_accepted"] == 1 and r["out_tokens"][0] == 1
    assert r["accept_ratio"][0] == pytest.approx(2 / 3, rel=1e-6)
    for u1 in (0.0, 0.5, 0.99):
        r = _single(oracle_mod, logits, q, [1], [0.9, u1])
        assert r["num_accepted"] == 0 and list(r["out_tokens"]) == [0, -1]


def test_greedy_is_sequential_argmax_decoding(oracle_mod):
    # tau = 0: accept while the draft equals argmax of its target row; the
    # emitted tokens are those of plain greedy decoding over the same rows.
    rng = np.random.default_rng(2)
    B, k, V = 400, 5, 11
    logits = rng.integers(-4, 5, size=(B, k + 1, V)).astype(np.float32)   # many ties
    best = np.argmax(logits, axis=-1)
    tokens = best[:, :k].copy()
    flip = rng.random((B, k)) < 0.25
    tokens[flip] = rng.integers(0, V, size=flip.sum())
    q = np.full((B, k, V), 1.0 / V, np.float32)
    u = rng.random((B, k + 1), dtype=np.float32)
    res = oracle_mod.accept(logits, q, tokens.astype(np.int32), u, np.zeros(B, np.float32))
    for b in range(B):
        n = 0
        while n < k and tokens[b, n] == best[b, n]:
            n += 1
        assert res["num_accepted"][b] == n
        expect = list(best[b, :n]) + [best[b, n]] + [-1] * (k - n)
        assert list(res["out_tokens"][b]) == expect
        assert np.isinf(res["margin"][b]).all()


def test_equal_distributions_accept_everything_and_draw_the_bonus(oracle_mod):
    rng = np.random.default_rng(3)
    B, k, V = 50, 4, 40
    logits = (3 * rng.standard_normal((B, k + 1, V))).astype(np.float32)
    p = softmax(logits.astype(np.float64), axis=-1)
    q = p[:, :k].astype(np.float32)
    tokens = rng.integers(0, V, size=(B, k)).astype(np.int32)
    u = (0.999 * rng.random((B, k + 1))).astype(np.float32)
    # keep clear of the fp32 rounding of q: require p/q comfortably above u
    res = oracle_mod.accept(logits, q, tokens, u, np.ones(B, np.float32))
    assert (res["num_accepted"] == k).all()
    for b in range(B):
        c = np.cumsum(p[b, k])
        assert res["out_tokens"][b, k] == int(np.searchsorted(c, u[b, k] * c[-1], side="right"))
        assert list(res["out_tokens"][b, :k]) == list(tokens[b])


def test_draft_on_a_zero_probability_token_is_rejected_and_resampled_from_p(oracle_mod):
    rng = np.random.default_rng(4)
    V = 30
    for trial in range(20):
        logits = (2 * rng.standard_normal((2, V))).astype(np.float32)
        x = int(rng.integers(0, V))
        logits[0, x] = -np.inf                       # p_0(x) = 0 exactly
        q = np.zeros((1, V), np.float32)
        q[0, x] = 1.0
        u = rng.random(2).astype(np.float32)
        r = _single(oracle_mod, logits, q, [x], u)
        assert r["num_accepted"] == 0
        p0 = softmax(logits[0].astype(np.float64))
        c = np.cumsum(p0)
        assert r["out_tokens"][0] == int(np.searchsorted(c, u[1] * c[-1], side="right"))


def test_draft_with_zero_draft_probability_is_accepted(oracle_mod):
    logits = np.zeros((2, 4), np.float32)
    q = np.array([[0.5, 0.5, 0.0, 0.0]], np.float32)
    r = _single(oracle_mod, logits, q, [2], [ONE_MINUS, 0.0])
    assert r["num_accepted"] == 1 and r["accept_ratio"][0] == 1.0


def test_temperature_divides_the_logits(oracle_mod):
    # softmax(L / 2) is softmax of the exactly halved logits at tau = 1.
    inp = make_accept_case(B=30, k=3, V=50, seed=5)
    a = oracle_mod.accept(inp.target_logits, inp.draft_probs, inp.draft_tokens, inp.uniforms,
                          np.full(30, 2.0, np.float32))
    b = oracle_mod.accept(inp.target_logits / np.float32(2), inp.draft_probs, inp.draft_tokens,
                          inp.uniforms, np.ones(30, np.float32))
    for key in ("num_accepted", "out_tokens"):
        np.testing.assert_array_equal(a[key], b[key])
    np.testing.assert_allclose(a["accept_ratio"], b["accept_ratio"], rtol=1e-14)


def _decide(oracle_mod, logits, q, x, u0, u1):
    r = _single(oracle_mod, logits, q, [x], [u0, u1])
    return int(r["num_accepted"]), int(r["out_tokens"][0])


def _bisect_f32(pred, lo=np.float32(0.0), hi=ONE_MINUS):
    """Smallest float32 u in (lo, hi] with pred(u) true, assuming pred is
    monotone (false then true) and pred(hi) is true."""
    lo_i = int(np.float32(lo).view(np.int32))
    hi_i = int(np.float32(hi).view(np.int32))
    while hi_i - lo_i > 1:
        mid = (lo_i + hi_i) // 2
        if pred(np.int32(mid).view(np.float32)):
            hi_i = mid
        else:
            lo_i = mid
    return float(np.int32(hi_i).view(np.float32))


@pytest.mark.parametrize("V,seed", [(2, 0), (3, 1), (5, 2), (8, 3)])
def test_output_distribution_equals_target_exactly(oracle_mod, V, seed):
    # Reconstruct, from the oracle's decisions alone, the probability of each
    # emitted token at position 0 when T'_1 ~ q and u0, u1 ~ U[0,1):
    # acceptance thresholds and residual CDF breakpoints are located by
    # bisection over the fp32 uniforms.  Speculative sampling's guarantee
    # (the emitted token is distributed as p) must hold to the resolution of
    # the fp32 grid.
    rng = np.random.default_rng(100 + seed)
    logits = (1.5 * rng.standard_normal((2, V))).astype(np.float32)
    q = softmax(rng.standard_normal(V) * 1.5).astype(np.float32)[None]
    p = softmax(logits[0].astype(np.float64))
    prob = np.zeros(V)
    for x in range(V):
        # acceptance region {u0 : accepted} is [0, a)
        if _decide(oracle_mod, logits, q, x, ONE_MINUS, 0.5)[0] == 1:
            a = 1.0
        else:
            a = _bisect_f32(lambda u: _decide(oracle_mod, logits, q, x, u, 0.5)[0] == 0)
        prob[x] += q[0, x] * a
        if a < 1.0:
            # residual draw: token as a function of u1 is a non-decreasing step
            prev = 0.0
            for y in range(V):
                if y == V - 1 or _decide(oracle_mod, logits, q, x, ONE_MINUS, ONE_MINUS)[1] <= y:
                    edge = 1.0
                else:
                    edge = _bisect_f32(
                        lambda u: _decide(oracle_mod, logits, q, x, ONE_MINUS, u)[1] > y)
                prob[y] += q[0, x] * (1 - a) * (edge - prev)
                prev = edge
    np.testing.assert_allclose(prob, p, rtol=0, atol=2e-6)


def _mc(oracle_mod, logits_rows, q_rows, trials, seed):
    k = q_rows.shape[0]
    V = q_rows.shape[1]
    rng = np.random.default_rng(seed)
    logits = np.broadcast_to(logits_rows, (trials, k + 1, V)).astype(np.float32)
    q = np.broadcast_to(q_rows, (trials, k, V)).astype(np.float32)
    qc = np.cumsum(q_rows.astype(np.float64), axis=-1)
    tokens = np.stack([np.minimum(np.searchsorted(qc[i], rng.random(trials) * qc[i, -1],
                                                  side="right"), V - 1) for i in range(k)],
                      axis=1).astype(np.int32)
    u = rng.random((trials, k + 1), dtype=np.float32)
    return oracle_mod.accept(logits, q, tokens, u, np.ones(trials, np.float32))


def test_monte_carlo_emitted_tokens_and_accepted_length(oracle_mod):
    # Independent rows, T'_i ~ q_i.  (1) the emitted token at position 0 is
    # distributed as p_0; (2) given n >= i it is distributed as p_i;
    # (3) P(n >= i) = prod_{j<i} beta_j with beta_j = sum_x min(p_j, q_j).
    rng = np.random.default_rng(7)
    k, V, trials = 3, 5, 400_000
    logits = (1.2 * rng.standard_normal((k + 1, V))).astype(np.float32)
    q_rows = softmax(logits[:k].astype(np.float64) + rng.standard_normal((k, V)),
                     axis=-1).astype(np.float32)
    res = _mc(oracle_mod, logits, q_rows, trials, seed=8)
    p = softmax(logits.astype(np.float64), axis=-1)
    n = res["num_accepted"]
    out = res["out_tokens"]
    alpha = 1e-4
    for i in range(k + 1):
        sel = n >= i
        obs = np.bincount(out[sel, i], minlength=V)
        assert chisquare(obs, p[i] * sel.sum()).pvalue > alpha, (i, obs, p[i] * sel.sum())
    beta = np.minimum(p[:k], q_rows.astype(np.float64)).sum(axis=-1)
    surv = np.concatenate([[1.0], np.cumprod(beta)])             # P(n >= i), i = 0..k
    law = np.append(surv[:-1] - surv[1:], surv[-1])              # P(n = i)
    obs = np.bincount(n, minlength=k + 1)
    assert chisquare(obs, law * trials).pvalue > alpha, (obs, law * trials)


def test_margins_are_reported_for_evaluated_decisions(oracle_mod):
    inp = make_accept_case(B=64, k=4, V=100, seed=9)
    res = oracle_mod.accept(inp.target_logits, inp.draft_probs, inp.draft_tokens, inp.uniforms,
                            inp.temperature)
    for b in range(64):
        j = res["num_accepted"][b]
        assert np.isfinite(res["margin"][b, :min(j + 1, 4)]).all()
        assert np.isinf(res["margin"][b, j + 1:4]).all()
        assert 0 <= res["margin"][b, 4] <= 1
        assert (res["out_tokens"][b, j + 1:] == -1).all()


def test_out_of_range_draft_token_is_an_error(oracle_mod):
    inp = make_accept_case(B=2, k=2, V=10, seed=10)
    tokens = inp.draft_tokens.copy()
    tokens[1, 1] = 10
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.accept(inp.target_logits, inp.draft_probs, tokens, inp.uniforms,
                          inp.temperature)
