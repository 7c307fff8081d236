"""Pins of the visual-compressor oracle (Sec. 3.2, Eq. 3):
F^_V = softmax(Q F_V^T) F_V per frame, softmax over the frame's tokens,
unscaled scores.

Each pin is fixed by the mathematics, not by re-running the formula: zero
queries give the plain mean of the tokens, one token gives itself, two
tokens give the logistic weight of the score difference, the output is a
convex combination, invariant under token permutations, equivariant under
query permutations, frames do not mix, and a query far more aligned with one
token than with the others returns that token (hard attention).
"""
import numpy as np
import pytest

from oracle import oracle as om
from paper_2505_12728_gb300.workloads import bf16_bits_to_f32, f32_to_bf16_bits


def bits(x):
    return f32_to_bf16_bits(np.asarray(x, np.float32))


def val(b):
    return bf16_bits_to_f32(b).astype(np.float64)


def rand_case(rng, F, N, C, d, q_std=0.3):
    q = bits(q_std * rng.standard_normal((C, d)))
    f = bits(rng.standard_normal((F, N, d)))
    return q, f


def test_zero_queries_give_the_token_mean():
    rng = np.random.default_rng(0)
    _, f = rand_case(rng, 2, 7, 3, 12)
    q = np.zeros((3, 12), np.uint16)
    out = om.visual_compress(q, f)
    for fr in range(2):
        np.testing.assert_allclose(out[fr], np.repeat(val(f[fr]).mean(0)[None], 3, 0), rtol=1e-13,
                                   atol=1e-14)


def test_one_token_is_returned_unchanged():
    rng = np.random.default_rng(1)
    q, f = rand_case(rng, 3, 1, 4, 9, q_std=2.0)
    out = om.visual_compress(q, f)
    for fr in range(3):
        np.testing.assert_array_equal(out[fr], np.repeat(val(f[fr]), 4, 0))


@pytest.mark.parametrize("a,b,x,y", [(1.0, 2.0, 0.5, -0.25), (3.0, -1.0, 1.5, 2.0), (0.5, 0.5, -4.0, 4.0)])
def test_two_tokens_follow_the_logistic_weight(a, b, x, y):
    # tokens [a, 0] and [0, b], query [x, y]: scores a*x and b*y (no scale),
    # weight of token 0 = 1 / (1 + exp(b*y - a*x))
    f = bits([[[a, 0.0], [0.0, b]]])
    q = bits([[x, y]])
    out = om.visual_compress(q, f)[0, 0]
    w = 1.0 / (1.0 + np.exp(b * y - a * x))
    np.testing.assert_allclose(out, [w * a, (1 - w) * b], rtol=1e-14, atol=1e-15)


def test_output_is_a_convex_combination_of_the_tokens():
    rng = np.random.default_rng(2)
    q, f = rand_case(rng, 2, 33, 5, 40, q_std=1.0)
    out = om.visual_compress(q, f)
    v = val(f)
    for fr in range(2):
        assert (out[fr] <= v[fr].max(0) + 1e-12).all() and (out[fr] >= v[fr].min(0) - 1e-12).all()


def test_token_permutation_invariance_and_query_equivariance():
    rng = np.random.default_rng(3)
    q, f = rand_case(rng, 1, 50, 6, 24, q_std=0.5)
    out = om.visual_compress(q, f)
    tp = rng.permutation(50)
    np.testing.assert_allclose(om.visual_compress(q, f[:, tp]), out, rtol=1e-12, atol=1e-14)
    qp = rng.permutation(6)
    np.testing.assert_allclose(om.visual_compress(q[qp], f), out[:, qp], rtol=1e-13, atol=1e-15)


def test_frames_are_compressed_independently():
    rng = np.random.default_rng(4)
    q, f = rand_case(rng, 3, 20, 4, 16, q_std=0.5)
    out = om.visual_compress(q, f)
    for fr in range(3):
        np.testing.assert_array_equal(om.visual_compress(q, f[fr:fr + 1])[0], out[fr])
    g = f.copy()
    g[0] = bits(rng.standard_normal((20, 16)))
    out2 = om.visual_compress(q, g)
    np.testing.assert_array_equal(out2[1:], out[1:])


def test_a_dominant_score_selects_its_token():
    # token k has feature 8 in its own column; the query weights that column
    # by 10: its score exceeds every other by >= 60, so the weight of every
    # other token is below e^-60
    N, d, k = 12, 16, 7
    f = np.zeros((1, N, d), np.float32)
    f[0, np.arange(N), np.arange(N)] = 1.0
    f[0, k, k] = 8.0
    q = np.zeros((1, d), np.float32)
    q[0, k] = 10.0
    out = om.visual_compress(bits(q), bits(f))[0, 0]
    np.testing.assert_allclose(out, f[0, k], atol=1e-24)


def test_shared_feature_column_does_not_change_weights():
    # every token has feature 1 in column 0: the query's column-0 weight adds
    # the same constant to all scores, which the softmax removes
    rng = np.random.default_rng(5)
    f = rng.standard_normal((1, 9, 6)).astype(np.float32)
    f[0, :, 0] = 1.0
    q = rng.standard_normal((2, 6)).astype(np.float32) * 0.5
    q2 = q.copy()
    q2[:, 0] += 3.0
    np.testing.assert_allclose(om.visual_compress(bits(q2), bits(f)),
                               om.visual_compress(bits(q), bits(f)), rtol=1e-12, atol=1e-14)


def test_invalid_shapes_raise():
    with pytest.raises(Exception):
        om.visual_compress(np.zeros((0, 4), np.uint16), np.zeros((1, 2, 4), np.uint16))
