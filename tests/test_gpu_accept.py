"""GPU parity of sf_accept against the fp64 oracle (C ABI path).

Accepted lengths, greedy tokens and resampled tokens must be bit-exact for
every sequence whose decisions the oracle does not place within 1e-6 of a
threshold or CDF boundary (given identical uniforms); acceptance ratios agree
to 2e-6.  A Monte-Carlo test checks the speculative-sampling guarantee on the
GPU's own outputs.
"""
import itertools

import numpy as np
import pytest
import torch
from scipy.special import softmax
from scipy.stats import chisquare

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import (AcceptInputs, WORKLOADS, make_accept_case,
                                              make_accept_inputs, workload)
from tests.gpu_helpers import (accept_to_device, compare_accept, oracle_accept, require_gpu,
                               run_accept)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _check(oracle_mod, inp, max_excluded_frac=0.02):
    n, toks, ratio = run_accept(inp)
    ref = oracle_accept(oracle_mod, inp)
    excluded = compare_accept(ref, n, toks, ratio)
    assert excluded <= max(1, max_excluded_frac * n.shape[0]), excluded
    return ref, n, toks


@pytest.mark.parametrize("name,mode", [("tiny", "greedy"), ("tiny", "sampling"),
                                       ("image7b", "sampling"), ("gqa", None), ("video", None)])
def test_named_workloads_match_oracle(oracle_mod, name, mode):
    _check(oracle_mod, make_accept_inputs(WORKLOADS[name], mode=mode))


@pytest.mark.parametrize("k", [2, 4, 8])
@pytest.mark.parametrize("mode", ["greedy", "sampling"])
def test_long_video_workload_matches_oracle(oracle_mod, k, mode):
    _check(oracle_mod, make_accept_inputs(workload("long", k=k), mode=mode))


@pytest.mark.parametrize("V", [32000, 152064, 5, 7, 1001, 32001])
def test_many_sequences_match_oracle(oracle_mod, V):
    B = 256 if V < 100000 else 48
    inp = make_accept_case(B, 4, V, seed=V, mode="alternate")
    _check(oracle_mod, inp)


@pytest.mark.parametrize("V", [32000, 152064])
def test_masked_target_logits_match_oracle(oracle_mod, V):
    # -inf target logits (a masked vocabulary) have probability 0 on both paths
    inp = make_accept_case(6, 4, V, seed=21, mode="alternate")
    inp.target_logits[:, :, ::3] = -np.inf
    inp.target_logits[:, :, 1] = 40.0  # keep a finite maximum
    ref, n, toks = _check(oracle_mod, inp)
    assert ((toks == -1) | (toks % 3 != 0)).all()


@pytest.mark.parametrize("mode", ["sampling", "greedy", "alternate"])
def test_vocabulary_beyond_the_single_kernel_path(oracle_mod, mode):
    # V above 16 slices of 2048 tokens: the two-kernel (statistics, draw) path
    _check(oracle_mod, make_accept_case(3, 4, 200003, seed=17, mode=mode))


@pytest.mark.parametrize("V", [300000, 300001])
@pytest.mark.parametrize("mode", ["sampling", "alternate"])
def test_vocabulary_beyond_256_segments(oracle_mod, V, mode):
    # more than 256 segments of 1024 tokens per row: the draw's last CTA
    # searches the segment sums block by block (one segment per thread
    # otherwise); V % 4 == 0 streams the logits by bulk copies, V % 4 != 0
    # through registers
    _check(oracle_mod, make_accept_case(2, 3, V, seed=V % 97, mode=mode))


def test_logits_not_16_byte_aligned(oracle_mod):
    # logits that start 4 bytes past a 16-byte boundary (V % 4 == 0): the
    # chunk kernel reads them through registers instead of bulk copies
    inp = make_accept_case(3, 4, 152064, seed=23, mode="alternate")
    dev = accept_to_device(inp)
    n_el = inp.target_logits.size
    big = torch.empty(n_el + 4, dtype=torch.float32, device="cuda")
    big[1:1 + n_el].copy_(torch.from_numpy(inp.target_logits.reshape(-1)).cuda())
    dev["target_logits"] = big[1:1 + n_el].view(inp.target_logits.shape)
    assert dev["target_logits"].data_ptr() % 16 == 4
    n, toks, ratio = run_accept(inp, dev=dev)
    ref = oracle_accept(oracle_mod, inp)
    assert compare_accept(ref, n, toks, ratio) <= 1


@pytest.mark.parametrize("V,k", [(2, 3), (3, 2), (5, 2), (5, 3)])
def test_brute_force_tiny_vocabularies(oracle_mod, V, k):
    # Every draft tuple in [0, V)^k, each with 64 uniform vectors drawn from
    # the 1/64 grid (cell midpoints), both modes; one fixed set of rows.
    rng = np.random.default_rng(V * 10 + k)
    logits_rows = (1.5 * rng.standard_normal((k + 1, V))).astype(np.float32)
    q_rows = softmax(logits_rows[:k].astype(np.float64) + rng.standard_normal((k, V)),
                     axis=-1).astype(np.float32)
    tuples = np.array(list(itertools.product(range(V), repeat=k)), np.int32)
    reps = 64
    B = len(tuples) * reps
    grid = (rng.integers(0, 64, size=(B, k + 1)) + 0.5) / 64
    for mode in ("sampling", "greedy"):
        inp = AcceptInputs(
            target_logits=np.ascontiguousarray(np.broadcast_to(logits_rows, (B, k + 1, V))),
            draft_probs=np.ascontiguousarray(np.broadcast_to(q_rows, (B, k, V))),
            draft_tokens=np.repeat(tuples, reps, axis=0),
            uniforms=grid.astype(np.float32),
            temperature=np.full(B, 1.0 if mode == "sampling" else 0.0, np.float32))
        # split into launches within the batch limit
        for s in range(0, B, 1024):
            sub = AcceptInputs(*(a[s:s + 1024] for a in (inp.target_logits, inp.draft_probs,
                                                          inp.draft_tokens, inp.uniforms,
                                                          inp.temperature)))
            _check(oracle_mod, sub)


def test_monte_carlo_output_distribution():
    # The emitted token at position i, given n >= i, is distributed as p_i,
    # and P(n >= i) = prod_{j<i} sum_x min(p_j, q_j); 2^20 trials in 1024
    # launches of 1024 sequences (the batch is the trial index).
    rng = np.random.default_rng(2026)
    k, V = 4, 5
    logits_rows = (1.2 * rng.standard_normal((k + 1, V))).astype(np.float32)
    q_rows = softmax(logits_rows[:k].astype(np.float64) + rng.standard_normal((k, V)),
                     axis=-1).astype(np.float32)
    p = softmax(logits_rows.astype(np.float64), axis=-1)
    Bl = 1024
    launches = 1024
    logits = torch.from_numpy(np.ascontiguousarray(np.broadcast_to(logits_rows, (Bl, k + 1, V)))).cuda()
    q = torch.from_numpy(np.ascontiguousarray(np.broadcast_to(q_rows, (Bl, k, V)))).cuda()
    temp = torch.ones(Bl, dtype=torch.float32, device="cuda")
    qc = np.cumsum(q_rows.astype(np.float64), axis=-1)
    ws = sfv.new_workspace(sfv.accept_workspace_size(Bl, k, V))
    ns, outs = [], []
    for it in range(launches):
        toks = np.stack([np.minimum(np.searchsorted(qc[i], rng.random(Bl) * qc[i, -1],
                                                    side="right"), V - 1) for i in range(k)],
                        axis=1).astype(np.int32)
        u = rng.random((Bl, k + 1), dtype=np.float32)
        n, o, _ = sfv.accept(logits, q, torch.from_numpy(toks).cuda(), torch.from_numpy(u).cuda(),
                             temp, workspace=ws)
        ns.append(n)
        outs.append(o)
    n = torch.cat(ns).cpu().numpy()
    out = torch.cat(outs).cpu().numpy()
    trials = n.shape[0]
    alpha = 1e-4
    for i in range(k + 1):
        sel = n >= i
        obs = np.bincount(out[sel, i], minlength=V)
        assert chisquare(obs, p[i] * sel.sum()).pvalue > alpha, (i, obs, p[i] * sel.sum())
    beta = np.minimum(p[:k], q_rows.astype(np.float64)).sum(axis=-1)
    surv = np.concatenate([[1.0], np.cumprod(beta)])
    law = np.append(surv[:-1] - surv[1:], surv[-1])
    obs = np.bincount(n, minlength=k + 1)
    assert chisquare(obs, law * trials).pvalue > alpha, (obs, law * trials)


def test_greedy_ties_take_the_lowest_token(oracle_mod):
    rng = np.random.default_rng(5)
    B, k, V = 300, 3, 64
    logits = rng.integers(-3, 3, size=(B, k + 1, V)).astype(np.float32)
    best = np.argmax(logits, axis=-1)
    tokens = best[:, :k].astype(np.int32).copy()
    flip = rng.random((B, k)) < 0.3
    tokens[flip] = rng.integers(0, V, size=flip.sum())
    inp = AcceptInputs(logits, np.full((B, k, V), 1.0 / V, np.float32), tokens,
                       rng.random((B, k + 1), dtype=np.float32), np.zeros(B, np.float32))
    ref, n, toks = _check(oracle_mod, inp, max_excluded_frac=0.0)
    assert (toks[np.arange(B), n] == best[np.arange(B), n]).all()


def test_equal_distributions_accept_all_and_use_the_bonus_row(oracle_mod):
    rng = np.random.default_rng(6)
    B, k, V = 64, 5, 4000
    logits = (3 * rng.standard_normal((B, k + 1, V))).astype(np.float32)
    q = softmax(logits[:, :k].astype(np.float64), axis=-1).astype(np.float32)
    tokens = rng.integers(0, V, size=(B, k)).astype(np.int32)
    u = (0.999 * rng.random((B, k + 1))).astype(np.float32)
    inp = AcceptInputs(logits, q, tokens, u, np.ones(B, np.float32))
    ref, n, toks = _check(oracle_mod, inp)
    assert (n == k).all()


@pytest.mark.parametrize("V", [32000, 152064])
def test_temperatures_other_than_one(oracle_mod, V):
    B = 128 if V < 100000 else 24
    inp = make_accept_case(B, 4, V, seed=7)
    inp.temperature = np.where(np.arange(B) % 3 == 0, 0.7, 1.3).astype(np.float32)
    _check(oracle_mod, inp)


def test_warp_runs_longer_than_32_chunks(oracle_mod):
    # 40 x 17 rows of 149 chunks: on a 152-SM part every warp of the chunk
    # kernel folds ~42 consecutive chunks, so runs cross rows mid-warp and
    # span more chunk records than a warp has lanes
    # (17 decisions per sequence: more of them fall within the oracle's margin)
    inp = make_accept_case(40, 16, 152064, seed=40, mode="alternate")
    _check(oracle_mod, inp, max_excluded_frac=0.1)


@pytest.mark.parametrize("B,k,V", [(1, 1, 32769), (1, 2, 40000), (3, 1, 33000), (2, 3, 65537)])
def test_fewer_chunks_than_warps_all_negative_logits(oracle_mod, B, k, V):
    # Few 1024-token chunks in all (B (k+1) ceil(V/1024) of 66 to 520): the
    # chunk kernel then runs one warp per chunk, and every row's run records
    # come from the warps that own its chunks.  Logits far below zero make
    # any stale or zero record visible: it would win the row maximum.
    ws = sfv.new_workspace(sfv.accept_workspace_size(B, k, V))
    for mode in ("greedy", "sampling"):
        inp = make_accept_case(B, k, V, seed=V + k, mode=mode)
        inp.target_logits -= np.float32(50.0)
        ref = oracle_accept(oracle_mod, inp)
        # twice on one workspace: the row and sequence tickets return to zero
        for _ in range(2):
            n, toks, ratio = run_accept(inp, workspace=ws)
            assert compare_accept(ref, n, toks, ratio) <= 1


def test_out_of_range_draft_token_is_flagged_and_rejected(oracle_mod):
    inp = make_accept_case(4, 3, 1000, seed=8)
    inp.draft_tokens[2, 1] = 5000
    dev = accept_to_device(inp)
    ws = sfv.new_workspace(sfv.accept_workspace_size(4, 3, 1000))
    n, toks, ratio = run_accept(inp, dev=dev, workspace=ws)
    assert sfv.read_device_status(ws) & sfv.SF_DEVICE_BAD_TOKEN
    assert n[2] <= 1


def test_repeated_calls_are_bit_identical():
    inp = make_accept_inputs(WORKLOADS["video"])
    dev = accept_to_device(inp)
    ws = sfv.new_workspace(sfv.accept_workspace_size(4, 8, 152064))
    a = run_accept(inp, dev=dev, workspace=ws)
    b = run_accept(inp, dev=dev, workspace=ws)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)
    assert sfv.read_device_status(ws) == 0


def test_kernel_launch_counts_follow_the_vocabulary():
    # one cluster kernel while a row fits 16 slices of 2048 tokens, else the
    # chunk kernel (statistics and decisions) and draw kernel
    assert sfv.accept_kernel_launches(1, 5, 32000) == 1
    assert sfv.accept_kernel_launches(4, 8, 32768) == 1
    assert sfv.accept_kernel_launches(4, 8, 32769) == 2
    assert sfv.accept_kernel_launches(8, 6, 152064) == 2


@pytest.mark.parametrize("V", [32000, 152064])
@pytest.mark.parametrize("mode", ["sampling", "alternate"])
def test_longest_draft_matches_oracle(oracle_mod, V, mode):
    # k = 16 drafts (the limit) on both acceptance paths
    inp = make_accept_case(8, 16, V, seed=[16, V], mode=mode)
    ref = oracle_accept(oracle_mod, inp)
    n, toks, ratio = run_accept(inp)
    excluded = compare_accept(ref, n, toks, ratio)
    assert excluded <= 1


@pytest.mark.parametrize("V,support", [
    # V = 40000: 512 tokens per warp, 4096 per CTA of the 16-CTA draw cluster
    (40000, [0, 511, 512, 4095, 4096, 20479, 20480, 39999]),
    # V = 152064: 1280 tokens per warp, 10240 per CTA
    (152064, [0, 1279, 1280, 10239, 10240, 81919, 81920, 152063]),
    # V % 4 != 0: the draw that searches segment sums after a ticket
    (40001, [0, 1023, 1024, 8191, 8192, 20480, 39999, 40000]),
])
def test_monte_carlo_large_vocabulary_draw(V, support):
    # The speculative-sampling guarantee at V > 32768 (statistics kernel and
    # a separate draw): the target has mass only on `support` (its tokens sit
    # on both sides of the draw's warp and CTA boundaries), the draft on an
    # overlapping set, so that the residual draw and the bonus draw both
    # matter.  2^15 trials in 64 launches of 512 sequences.
    rng = np.random.default_rng(V)
    k = 2
    sup = np.array(support)
    dsup = np.array(sorted(set(support[::2]) | {support[3], support[5]}))
    logits_rows = np.full((k + 1, V), -np.inf, np.float32)
    logits_rows[:, sup] = rng.standard_normal((k + 1, len(sup))).astype(np.float32)
    q_rows = np.zeros((k, V), np.float32)
    q_rows[:, dsup] = softmax(rng.standard_normal((k, len(dsup))), axis=-1).astype(np.float32)
    p = softmax(logits_rows.astype(np.float64), axis=-1)
    Bl, launches = 512, 64
    logits = torch.from_numpy(logits_rows).cuda().unsqueeze(0).expand(Bl, k + 1, V).contiguous()
    q = torch.from_numpy(q_rows).cuda().unsqueeze(0).expand(Bl, k, V).contiguous()
    temp = torch.ones(Bl, dtype=torch.float32, device="cuda")
    qd = q_rows[:, dsup].astype(np.float64)
    qc = np.cumsum(qd, axis=-1)
    ws = sfv.new_workspace(sfv.accept_workspace_size(Bl, k, V))
    ns, outs = [], []
    for _ in range(launches):
        toks = np.stack([dsup[np.minimum(np.searchsorted(qc[i], rng.random(Bl) * qc[i, -1],
                                                         side="right"), len(dsup) - 1)]
                         for i in range(k)], axis=1).astype(np.int32)
        u = rng.random((Bl, k + 1), dtype=np.float32)
        n, o, _ = sfv.accept(logits, q, torch.from_numpy(toks).cuda(), torch.from_numpy(u).cuda(),
                             temp, workspace=ws)
        ns.append(n)
        outs.append(o)
    assert sfv.read_device_status(ws) == 0
    n = torch.cat(ns).cpu().numpy()
    out = torch.cat(outs).cpu().numpy()
    trials = n.shape[0]
    alpha = 1e-4
    for i in range(k + 1):
        sel = n >= i
        emitted = out[sel, i]
        assert np.isin(emitted, sup).all(), np.setdiff1d(emitted, sup)
        obs = np.array([(emitted == t).sum() for t in sup])
        assert chisquare(obs, p[i, sup] * sel.sum()).pvalue > alpha, (i, obs, p[i, sup] * sel.sum())
    beta = np.minimum(p[:k], q_rows.astype(np.float64)).sum(axis=-1)
    surv = np.concatenate([[1.0], np.cumprod(beta)])
    law = np.append(surv[:-1] - surv[1:], surv[-1])
    obs = np.bincount(n, minlength=k + 1)
    assert chisquare(obs, law * trials).pvalue > alpha, (obs, law * trials)


@pytest.mark.parametrize("V", [40000, 40001, 152064])
def test_residual_without_mass_draws_from_the_target(oracle_mod, V):
    # q = 1.001 p everywhere: the residual max(0, p - q) is exactly zero, and
    # u_0 = 0.9995 > p/q rejects the first draft (by a relative margin of
    # 5e-4), so the token comes from p_0 itself on both sides (logits with a
    # wide spread, so that the draw's CDF steps are large against the
    # oracle's 1e-6 margin)
    rng = np.random.default_rng(V + 1)
    B, k = 8, 2
    logits = (6.0 * rng.standard_normal((B, k + 1, V))).astype(np.float32)
    p = softmax(logits.astype(np.float64), axis=-1)
    q = (1.001 * p[:, :k]).astype(np.float32)
    tokens = np.argmax(q, axis=-1).astype(np.int32)
    u = rng.random((B, k + 1), dtype=np.float32)
    u[:, 0] = 0.9995
    inp = AcceptInputs(logits, q, tokens, u, np.ones(B, np.float32))
    ref, n, toks = _check(oracle_mod, inp, max_excluded_frac=0.0)
    assert (n == 0).all()
