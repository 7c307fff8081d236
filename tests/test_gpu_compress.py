"""GPU parity of the visual compressor (Sec. 3.2, Eq. 3) against the fp64
oracle, through the C ABI.

Tolerance, derived from the arithmetic: the scores are fp32 sums of exact
bf16 products (relative error ~1e-5 of the weights); the weights exp(s - max)
are rounded to bf16 (relative 2^-9 each) and the output is their exact
convex combination divided by the sum of the rounded weights, so it moves by
at most 2^-8 * max_n |F_V[n][j] - out[j]|; the bf16 output adds 2^-9 |out[j]|.
"""
import numpy as np
import pytest
import torch

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import (COMPRESS_SHAPES, bf16_bits_to_f32,
                                              make_compress_case)
from tests.gpu_helpers import bf16_tensor, require_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def run(queries, features):
    ws = sfv.new_workspace(sfv.visual_compress_workspace_size(*features.shape[:2], *queries.shape))
    out = sfv.visual_compress(bf16_tensor(queries), bf16_tensor(features), workspace=ws)
    torch.cuda.synchronize()
    assert sfv.read_device_status(ws) == 0
    return out.float().cpu().numpy()


def bound(features, ref):
    v = bf16_bits_to_f32(features).astype(np.float64)          # [F][N][d]
    # max_n |v[n][j] - out[c][j]| from the per-column extremes of the frame
    vmax, vmin = v.max(axis=1)[:, None, :], v.min(axis=1)[:, None, :]
    spread = np.maximum(vmax - ref, ref - vmin)                   # [F][C][d]
    return 2.0 ** -8 * spread + 2.0 ** -9 * np.abs(ref) + 1e-4


def check(oracle_mod, queries, features):
    got = run(queries, features)
    ref = oracle_mod.visual_compress(queries, features)
    lim = bound(features, ref)
    err = np.abs(got - ref)
    worst = np.unravel_index(np.argmax(err / lim), err.shape)
    assert np.isfinite(got).all()
    assert (err <= lim).all(), f"max err/bound {(err / lim).max():.3f} at {worst}: {got[worst]} vs {ref[worst]}"
    return got, ref


@pytest.mark.parametrize("F,N,C,d", [
    (1, 16, 8, 128),        # one MMA step
    (3, 100, 36, 256),      # ragged N (Npad 112), QwenVL C
    (2, 37, 5, 128),        # N % 4 != 0: scalar score reads
    (2, 768, 128, 128),     # the largest N and C
    (4, 1, 3, 384),         # one token per frame: out = that token
    (9, 324, 36, 640),      # QwenVL images, 9 frames
])
def test_compressor_matches_oracle(oracle_mod, F, N, C, d):
    q, f = make_compress_case(F, N, C, d, seed=[F, N, C, d])
    got, ref = check(oracle_mod, q, f)
    if N == 1:
        np.testing.assert_array_equal(got, np.repeat(bf16_bits_to_f32(f), C, axis=1))


@pytest.mark.parametrize("name", ["image7b", "gqa"])
def test_named_workload_compressor_matches_oracle(oracle_mod, name):
    F, N, C, d = COMPRESS_SHAPES[name]
    q, f = make_compress_case(F, N, C, d, seed=[1, F])
    check(oracle_mod, q, f)


def test_video_workload_sampled_frames(oracle_mod):
    # 128 frames of 144 tokens at d 3584: the GPU runs all of them; the oracle
    # checks 6 sampled frames
    F, N, C, d = COMPRESS_SHAPES["video"]
    q, f = make_compress_case(F, N, C, d, seed=2)
    got = run(q, f)
    frames = np.random.default_rng(0).choice(F, 6, replace=False)
    ref = oracle_mod.visual_compress(q, f[frames])
    assert (np.abs(got[frames] - ref) <= bound(f[frames], ref)).all()


def test_zero_queries_average_the_tokens():
    F, N, C, d = 2, 50, 4, 256
    _, f = make_compress_case(F, N, C, d, seed=3)
    got = run(np.zeros((C, d), np.uint16), f)
    mean = bf16_bits_to_f32(f).astype(np.float64).mean(axis=1)
    assert np.abs(got - mean[:, None, :]).max() <= 2.0 ** -8 * 4 + 1e-3


def test_sharp_scores_select_one_token():
    # every query is 64x one token's features: its weight dominates
    F, N, C, d = 1, 64, 8, 128
    _, f = make_compress_case(F, N, C, d, seed=4)
    v = bf16_bits_to_f32(f).astype(np.float32)
    pick = np.arange(C) * 7
    from paper_2505_12728_gb300.workloads import f32_to_bf16_bits
    q = f32_to_bf16_bits(v[0, pick])
    got = run(q, f)
    # the query of token t scores |v_t|^2 ~ 128 on it and ~N(0, 128) on the
    # others: the weight of t dominates unless another token comes close
    ref_w = v[0] @ v[0, pick].T                          # [N][C]
    gap = ref_w[pick, np.arange(C)] - np.sort(ref_w, axis=0)[-2]
    sharp = gap > 30
    assert sharp.sum() >= C // 2
    assert np.abs(got[0][sharp] - v[0, pick][sharp]).max() <= 0.05


def test_compressor_is_deterministic():
    q, f = make_compress_case(3, 200, 20, 512, seed=5)
    a = run(q, f)
    b = run(q, f)
    assert np.array_equal(a, b)


def test_compressor_invalid_arguments():
    lib = sfv.load_library()
    q = torch.zeros((4, 128), dtype=torch.bfloat16, device="cuda")
    f = torch.zeros((1, 8, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((1, 4, 128), dtype=torch.bfloat16, device="cuda")
    ws = sfv.new_workspace(sfv.visual_compress_workspace_size(1, 8, 4, 128))
    P = lambda t: t.data_ptr()
    n = ws.numel()
    assert lib.sf_visual_compress(P(q), P(f), 1, 8, 4, 128, P(out), P(ws), n, None) == 0
    assert lib.sf_visual_compress(P(q), P(f), 1, 769, 4, 128, P(out), P(ws), n, None) == 1
    assert lib.sf_visual_compress(P(q), P(f), 1, 8, 129, 128, P(out), P(ws), n, None) == 1
    assert lib.sf_visual_compress(P(q), P(f), 1, 8, 4, 96, P(out), P(ws), n, None) == 1
    assert lib.sf_visual_compress(P(q), P(f), 0, 8, 4, 128, P(out), P(ws), n, None) == 1
    assert lib.sf_visual_compress(P(q), P(f), 1, 8, 4, 128, P(out), P(ws), 16, None) == 4
    assert lib.sf_visual_compress_workspace_size(1, 769, 4, 128) == 0
    torch.cuda.synchronize()
