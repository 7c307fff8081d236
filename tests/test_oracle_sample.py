"""Pins of the draft-tail oracle: LM-head logits and the sampling of T'.

Algorithm 1 ends with P'_i = LM-head(F'_{M+i}) and T'_i ~ Categorical(P'_i).
The sampler is pinned against an independent softmax (scipy), hand-worked
cases, the exact output distribution recovered by bisection over the
uniform, a Monte Carlo check, and greedy ties; the logits against a
brute-force triple loop and unit-vector weights.
"""
import numpy as np
import pytest
from scipy.special import softmax

from oracle import oracle as om
from paper_2505_12728_gb300.workloads import bf16_bits_to_f32, f32_to_bf16_bits


def test_probs_are_the_tempered_softmax():
    rng = np.random.default_rng(0)
    logits = (rng.standard_normal((6, 257)) * 3).astype(np.float32)
    for tau in (1.0, 0.5, 2.0):
        p, _, _ = om.sample(logits, rng.random(6).astype(np.float32), np.full(6, tau, np.float32))
        np.testing.assert_allclose(p, softmax(logits.astype(np.float64) / tau, axis=1), rtol=1e-12,
                                   atol=1e-15)


def test_hand_worked_draws():
    logits = np.array([[0.0, 1.0, 2.0]] * 4, np.float32)
    # softmax = [0.0900, 0.2447, 0.6652]; CDF = [0.0900, 0.3348, 1.0]
    u = np.array([0.05, 0.2, 0.5, 0.999], np.float32)
    _, tok, mg = om.sample(logits, u, np.ones(4, np.float32))
    assert tok.tolist() == [0, 1, 2, 2]
    assert abs(mg[2] - (0.5 - 0.33475904)) < 1e-6


def test_draw_at_a_boundary_goes_to_the_next_token():
    # two equal logits: C(0) / S = 0.5 exactly; u = 0.5 is not < 0.5, so x = 1
    _, tok, mg = om.sample(np.array([[0.0, 0.0]], np.float32), np.array([0.5], np.float32),
                           np.ones(1, np.float32))
    assert tok[0] == 1 and mg[0] == 0.0


def test_greedy_is_first_argmax_with_one_hot_probs():
    logits = np.array([[1.0, 3.0, 3.0, -2.0], [5.0, 4.0, 5.0, 5.0]], np.float32)
    p, tok, mg = om.sample(logits, np.array([0.9, 0.1], np.float32), np.array([0.0, -1.0], np.float32))
    assert tok.tolist() == [1, 0]
    assert p.tolist() == [[0, 1, 0, 0], [1, 0, 0, 0]]
    assert mg.tolist() == [0.0, 0.0]


def test_output_distribution_is_exact():
    # the token is a non-decreasing step function of u: find every step by
    # bisection over fp32 uniforms; the step widths are the probabilities
    logits = np.array([[0.3, -1.2, 2.0, 0.7, 0.0]], np.float32)
    tau = np.ones(1, np.float32)
    probs = softmax(logits.astype(np.float64)[0])

    def tok(u):
        return int(om.sample(logits, np.array([u], np.float32), tau)[1][0])

    edges = []
    for x in range(1, 5):
        lo, hi = np.float32(0.0), np.float32(1.0 - 2 ** -24)
        while np.nextafter(lo, np.float32(1)) < hi:
            mid = np.float32((np.float64(lo) + np.float64(hi)) / 2)
            if mid == lo or mid == hi:
                break
            if tok(float(mid)) >= x:
                hi = mid
            else:
                lo = mid
        edges.append(float(hi))
    widths = np.diff([0.0] + edges + [1.0])
    np.testing.assert_allclose(widths, probs, atol=1e-6)


def test_monte_carlo_frequencies():
    rng = np.random.default_rng(3)
    V, n = 7, 200_000
    logits = np.tile((rng.standard_normal(V) * 2).astype(np.float32), (n, 1))
    u = rng.random(n).astype(np.float32)
    p, tok, _ = om.sample(logits, u, np.full(n, 1.5, np.float32))
    freq = np.bincount(tok, minlength=V) / n
    sd = np.sqrt(p[0] * (1 - p[0]) / n)
    assert np.all(np.abs(freq - p[0]) < 5 * sd + 1e-9)


def test_temperature_scales_the_logits():
    logits = np.array([[0.0, 2.0, 4.0]], np.float32)
    p2, _, _ = om.sample(logits, np.array([0.5], np.float32), np.array([2.0], np.float32))
    p1, _, _ = om.sample(logits / 2, np.array([0.5], np.float32), np.array([1.0], np.float32))
    np.testing.assert_allclose(p2, p1, rtol=1e-12)


def test_lm_head_logits_brute_force_and_unit_vectors():
    rng = np.random.default_rng(4)
    h = f32_to_bf16_bits(rng.standard_normal((3, 5)).astype(np.float32))
    w = f32_to_bf16_bits(rng.standard_normal((4, 5)).astype(np.float32))
    got = om.lm_head_logits(h, w)
    hf, wf = bf16_bits_to_f32(h).astype(np.float64), bf16_bits_to_f32(w).astype(np.float64)
    for r in range(3):
        for v in range(4):
            assert abs(got[r, v] - sum(hf[r, c] * wf[v, c] for c in range(5))) < 1e-12
    # weights = 2 x unit vectors: logits are twice the hidden components
    eye = f32_to_bf16_bits((2 * np.eye(5)).astype(np.float32))
    np.testing.assert_array_equal(om.lm_head_logits(h, eye), 2 * hf)
