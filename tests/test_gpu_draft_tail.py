"""GPU parity of the draft-distribution tail (Algorithm 1: the frozen LM
head, then P' = softmax(logits / tau) and T' ~ Categorical(P')) against the
fp64 oracle, through the C ABI.

Tolerances, derived from the arithmetic:
  * LM head: bf16 products are exact in fp32 and the tensor cores accumulate
    in fp32, about K/16 roundings of partial sums; |error| <= sqrt(K) * 2^-24 *
    sum_j |h_j w_j| is well above that (the rounding errors add like a random
    walk) and far below the effect of one dropped product or 16-column step.
  * Sampler on identical fp32 logits: P' to 2e-6 relative (fp32 exp of a
    float-float argument, ~2 ulp, times an fp32 reciprocal of the
    float-float sum); T' bit-exact wherever the oracle's CDF boundary
    distance (margin) is >= 1e-6.
  * Fused path (projection + sampling): on small-integer inputs scaled by a
    power of two every partial sum is exact in fp32, so the GPU's logits
    must equal the oracle's bit for bit and the samples are compared as
    above; on N(0,1)-scale inputs the fused path must agree with the
    stand-alone sampler run on its own logits.
"""
import numpy as np
import pytest
import torch

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import (WORKLOADS, bf16_bits_to_f32,
                                              make_draft_tail_case, make_draft_tail_inputs,
                                              make_sample_case)
from tests.gpu_helpers import MARGIN, bf16_tensor, require_gpu

pytestmark = pytest.mark.gpu

PROB_RTOL = 2e-6
PROB_ATOL = 1e-37


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def lm_bound(hidden_bits, weight_bits):
    """Per-logit error bound sqrt(K) 2^-24 sum_j |h_j w_j| (float64 [R][V])."""
    h = np.abs(bf16_bits_to_f32(hidden_bits).astype(np.float64))
    w = np.abs(bf16_bits_to_f32(weight_bits).astype(np.float64))
    K = h.shape[1]
    return np.sqrt(K) * 2.0 ** -24 * (h @ w.T) + 1e-7


def run_sample(logits, uniforms, temperature):
    d = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (logits, uniforms, temperature)]
    probs, tokens = sfv.sample(*d)
    torch.cuda.synchronize()
    return probs.cpu().numpy(), tokens.cpu().numpy()


def run_fused(case):
    h, w = bf16_tensor(case.hidden), bf16_tensor(case.weight)
    u = torch.from_numpy(case.uniforms).cuda()
    t = torch.from_numpy(case.temperature).cuda()
    ws = sfv.new_workspace(sfv.draft_tail_workspace_size(*case.hidden.shape[:1], case.weight.shape[0]))
    logits, probs, tokens = sfv.draft_sample(h, w, u, t, workspace=ws)
    torch.cuda.synchronize()
    assert sfv.read_device_status(ws) == 0
    return logits.cpu().numpy(), probs.cpu().numpy(), tokens.cpu().numpy()


def check_sampler(oracle_mod, logits, uniforms, temperature, probs, tokens):
    ref_p, ref_t, margin = oracle_mod.sample(logits, uniforms, temperature)
    assert tokens.dtype == np.int32 and ((tokens >= 0) & (tokens < logits.shape[1])).all()
    decided = margin >= MARGIN
    greedy = ~(temperature > 0)
    decided |= greedy  # the argmax of identical fp32 values is exact
    bad = np.nonzero(decided & (tokens != ref_t))[0]
    assert bad.size == 0, f"rows {bad[:8]}: gpu {tokens[bad[:8]]} oracle {ref_t[bad[:8]]}"
    err = np.abs(probs.astype(np.float64) - ref_p)
    lim = PROB_RTOL * ref_p + PROB_ATOL
    worst = np.unravel_index(np.argmax(err - lim), err.shape)
    assert (err <= lim).all(), f"probs at {worst}: {probs[worst]} vs {ref_p[worst]}"
    # every drawn token has positive probability
    assert (probs[np.arange(len(tokens)), tokens] > 0).all()
    return int((~decided).sum())


# --------------------------------------------------------------------------- #
# LM head                                                                     #
# --------------------------------------------------------------------------- #
@pytest.mark.parametrize("R,Hd,V", [
    (1, 64, 128),        # one tile, one chunk
    (5, 4096, 32000),    # LLaVA draft rows (k = 5)
    (17, 200, 1000),     # ragged: hidden not a multiple of 64, V not of 128, NP = 32
    (48, 3584, 4099),    # 48 rows (B8 x k6), a ragged last tile
    (128, 512, 20000),   # B16 x k8 rows
    (256, 256, 3000),    # the largest N
    (3, 8, 300),         # the smallest hidden size (one zero-filled chunk)
])
def test_lm_head_matches_oracle(oracle_mod, R, Hd, V):
    case = make_draft_tail_case(R, Hd, V, seed=[R, Hd, V])
    logits = sfv.lm_head(bf16_tensor(case.hidden), bf16_tensor(case.weight))
    torch.cuda.synchronize()
    got = logits.cpu().numpy().astype(np.float64)
    ref = oracle_mod.lm_head_logits(case.hidden, case.weight)
    bound = lm_bound(case.hidden, case.weight)
    ratio = np.abs(got - ref) / bound
    assert np.isfinite(got).all()
    assert ratio.max() <= 1.0, f"max error / bound = {ratio.max()} at {np.unravel_index(ratio.argmax(), ratio.shape)}"


@pytest.mark.parametrize("R,Hd,V", [(5, 4096, 32000), (33, 3584, 5000), (200, 96, 700)])
def test_lm_head_exact_on_small_integer_inputs(oracle_mod, R, Hd, V):
    # exactly representable partial sums: the logits equal the oracle's
    case = make_draft_tail_case(R, Hd, V, seed=[R, 1], exact=True)
    logits = sfv.lm_head(bf16_tensor(case.hidden), bf16_tensor(case.weight))
    torch.cuda.synchronize()
    assert np.array_equal(logits.cpu().numpy().astype(np.float64),
                          oracle_mod.lm_head_logits(case.hidden, case.weight))


def test_lm_head_is_deterministic():
    case = make_draft_tail_case(40, 1024, 9000, seed=7)
    h, w = bf16_tensor(case.hidden), bf16_tensor(case.weight)
    a = sfv.lm_head(h, w)
    b = sfv.lm_head(h, w)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_lm_head_unit_rows_select_weight_columns():
    # hidden row r = e_{j_r} (bf16 1.0): logits[r][v] = w[v][j_r] exactly
    R, Hd, V = 16, 384, 2500
    case = make_draft_tail_case(R, Hd, V, seed=11)
    cols = np.random.default_rng(3).choice(Hd, R, replace=False)
    hidden = np.zeros((R, Hd), np.uint16)
    hidden[np.arange(R), cols] = 0x3F80
    logits = sfv.lm_head(bf16_tensor(hidden), bf16_tensor(case.weight))
    torch.cuda.synchronize()
    want = bf16_bits_to_f32(case.weight)[:, cols].T
    assert np.array_equal(logits.cpu().numpy(), want)


# --------------------------------------------------------------------------- #
# sampler on given logits                                                     #
# --------------------------------------------------------------------------- #
@pytest.mark.parametrize("V", [1, 3, 1000, 2048, 4097, 32000, 152064])
def test_sample_matches_oracle(oracle_mod, V):
    R = 12
    temp = np.array([1, 1, 0.7, 2.0, 0, 1, 0.05, 1, -1, 1.3, 1, 0], np.float32)
    logits, u, _ = make_sample_case(R, V, seed=V)
    u[0] = 0.0
    u[1] = np.float32(1 - 2 ** -24)
    probs, tokens = run_sample(logits, u, temp)
    check_sampler(oracle_mod, logits, u, temp, probs, tokens)


def test_sample_many_rows_and_unaligned_vocabulary(oracle_mod):
    R, V = 300, 5001  # V % 4 != 0: the scalar path
    logits, u, _ = make_sample_case(R, V, seed=99, logit_std=5.0)
    temp = np.where(np.arange(R) % 5 == 0, 0.0, 1.0 + (np.arange(R) % 3) * 0.25).astype(np.float32)
    probs, tokens = run_sample(logits, u, temp)
    excluded = check_sampler(oracle_mod, logits, u, temp, probs, tokens)
    assert excluded <= 3


def test_sample_masked_tokens_and_ties(oracle_mod):
    R, V = 6, 7000
    logits, u, temp = make_sample_case(R, V, seed=5)
    logits[0, :6990] = -np.inf           # only the last ten tokens are allowed
    logits[1, ::2] = -np.inf
    logits[2, :] = 1.5                   # all equal: uniform P', greedy picks token 0
    logits[3, 100] = logits[3, 200] = logits[3].max() + 4.0  # a tie for the argmax
    temp[2] = 0.0
    temp[3] = 0.0
    probs, tokens = run_sample(logits, u, temp)
    check_sampler(oracle_mod, logits, u, temp, probs, tokens)
    assert tokens[2] == 0 and tokens[3] == 100
    assert tokens[0] >= 6990 and tokens[1] % 2 == 1
    assert (probs[0, :6990] == 0).all() and (probs[1, ::2] == 0).all()


def test_sample_distribution_follows_probs():
    # many rows of the same logits with fresh uniforms: token frequencies
    # follow P' (chi-square on the GPU's own outputs)
    from scipy.stats import chisquare
    V, R = 40, 60000
    base = np.random.default_rng(1).standard_normal(V).astype(np.float32)
    logits = np.repeat(base[None], R, axis=0)
    u = np.random.default_rng(2).random(R, dtype=np.float32)
    temp = np.full(R, 0.8, np.float32)
    probs, tokens = run_sample(logits, u, temp)
    counts = np.bincount(tokens, minlength=V)
    expected = probs[0].astype(np.float64) * R
    keep = expected > 5
    stat = chisquare(counts[keep], expected[keep] / expected[keep].sum() * counts[keep].sum())
    assert stat.pvalue > 1e-4


# --------------------------------------------------------------------------- #
# fused projection + sampling                                                 #
# --------------------------------------------------------------------------- #
# With small-integer inputs (make_draft_tail_case(exact=True)) every fp32
# accumulation order gives the exact logits, so the GPU's logits must equal
# the oracle's bit for bit and the sampled tokens are compared exactly (away
# from 1e-6 of a CDF boundary), like the sampler on identical logits.
def check_fused(oracle_mod, case, logits, probs, tokens):
    ref_logits = oracle_mod.lm_head_logits(case.hidden, case.weight)
    assert np.array_equal(logits.astype(np.float64), ref_logits)
    return check_sampler(oracle_mod, ref_logits.astype(np.float32), case.uniforms,
                         case.temperature, probs, tokens)


@pytest.mark.parametrize("R,Hd,V,mode", [
    (5, 4096, 32000, "sampling"),
    (12, 512, 1000, "mixed"),
    (48, 1024, 6000, "mixed"),
    (1, 64, 7, "sampling"),
    (130, 256, 3001, "mixed"),
    (256, 128, 2000, "mixed"),
])
def test_draft_sample_matches_oracle(oracle_mod, R, Hd, V, mode):
    temp = np.ones(R, np.float32) if mode == "sampling" else \
        np.where(np.arange(R) % 3 == 0, 0.0, 0.6 + 0.2 * (np.arange(R) % 4)).astype(np.float32)
    case = make_draft_tail_case(R, Hd, V, seed=[R, V, 3], temperature=temp, exact=True)
    logits, probs, tokens = run_fused(case)
    excluded = check_fused(oracle_mod, case, logits, probs, tokens)
    assert excluded <= max(2, R // 5)


def test_draft_sample_real_valued_inputs():
    # N(0,1)-scale inputs: the logits are checked by the LM-head bound; the
    # fused statistics and the stand-alone sampler give the same P' (to
    # rounding) and, away from boundaries, the same T'
    case = make_draft_tail_case(64, 1024, 12345, seed=4,
                                temperature=np.linspace(0.0, 2.0, 64).astype(np.float32))
    logits, probs, tokens = run_fused(case)
    p2, t2 = run_sample(logits, case.uniforms, case.temperature)
    assert np.allclose(probs, p2, rtol=4e-6, atol=1e-37)
    assert (tokens == t2).mean() >= 0.95
    s = probs.astype(np.float64).sum(axis=1)
    assert np.abs(s - 1).max() < 1e-5
    assert (probs[np.arange(64), tokens] > 0).all()


@pytest.mark.parametrize("name", ["image7b", "gqa"])
def test_named_workload_draft_tail_matches_oracle(oracle_mod, name):
    wl = WORKLOADS[name]
    case = make_draft_tail_inputs(wl, exact=True)
    logits, probs, tokens = run_fused(case)
    excluded = check_fused(oracle_mod, case, logits, probs, tokens)
    assert excluded <= max(2, case.hidden.shape[0] // 5)


def test_long_workload_sampled_rows(oracle_mod):
    # B16 x k8 = 128 rows over the 152064 x 3584 LM head: the GPU runs the
    # full launch; the oracle checks 12 sampled rows end to end
    wl = WORKLOADS["long"]
    case = make_draft_tail_inputs(wl, exact=True)
    logits, probs, tokens = run_fused(case)
    rows = np.sort(np.random.default_rng(0).choice(case.hidden.shape[0], 12, replace=False))
    ref = np.concatenate([oracle_mod.lm_head_logits(case.hidden[rows], case.weight[v:v + 16384])
                          for v in range(0, wl.V, 16384)], axis=1)
    assert np.array_equal(logits[rows].astype(np.float64), ref)
    check_sampler(oracle_mod, ref.astype(np.float32), case.uniforms[rows],
                  case.temperature[rows], probs[rows], tokens[rows])
    s = probs.astype(np.float64).sum(axis=1)
    assert np.abs(s - 1).max() < 1e-5


# --------------------------------------------------------------------------- #
# argument checks                                                             #
# --------------------------------------------------------------------------- #
def test_draft_tail_invalid_arguments_are_rejected():
    case = make_draft_tail_case(4, 64, 100, seed=0)
    h, w = bf16_tensor(case.hidden), bf16_tensor(case.weight)
    lib = sfv.load_library()
    out = torch.empty((4, 100), dtype=torch.float32, device="cuda")
    ws = sfv.new_workspace(sfv.draft_tail_workspace_size(4, 100))
    P = lambda t: None if t is None else t.data_ptr()
    assert lib.sf_lm_head(P(h), P(w), 0, 64, 100, P(out), P(ws), ws.numel(), None) == 1
    assert lib.sf_lm_head(P(h), P(w), 257, 64, 100, P(out), P(ws), ws.numel(), None) == 1
    assert lib.sf_lm_head(P(h), P(w), 4, 60, 100, P(out), P(ws), ws.numel(), None) == 1
    assert lib.sf_lm_head(P(h) + 2, P(w), 4, 64, 100, P(out), P(ws), ws.numel(), None) == 1
    assert lib.sf_lm_head(P(h), P(w), 4, 64, 100, P(out), None, 0, None) == 4
    u = torch.zeros(4, dtype=torch.float32, device="cuda")
    tok = torch.empty(4, dtype=torch.int32, device="cuda")
    assert lib.sf_sample(P(out), P(u), P(u), 4, 100, P(out), P(tok), P(ws), 16, None) == 4
    assert lib.sf_sample(P(out), P(u), None, 4, 100, P(out), P(tok), P(ws), ws.numel(), None) == 1
    assert lib.sf_draft_tail_workspace_size(0, 100) == 0
    torch.cuda.synchronize()
