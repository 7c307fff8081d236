"""GPU parity of the fused target LM head + acceptance (sf_verify_lm_head_accept)
against the fp64 oracle.

The hidden states and LM-head weights are small integers (weights scaled by a
power of two): every fp32 partial sum is exact, so the GPU's logits must equal
the oracle's LM-head logits bit for bit, and the accepted lengths and tokens
are then compared exactly with the oracle's rule on those logits (excluding
decisions within 1e-6 of a threshold or CDF boundary, as for sf_accept).
The draft distribution q is the softmax of the target logits plus noise.
"""
import numpy as np
import pytest
import torch
from scipy.special import softmax

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import (AcceptInputs, HIDDEN_SIZES, WORKLOADS,
                                              make_draft_tail_case, temperatures)
from tests.gpu_helpers import bf16_tensor, compare_accept, oracle_accept, require_gpu, run_accept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def make_case(oracle_mod, B, k, V, d, seed, mode="sampling", sharpness=1.0):
    # exact small-integer hidden states [B*(k+1)][d] and weights [V][d]
    dt = make_draft_tail_case(B * (k + 1), d, V, seed=seed, exact=True)
    logits = oracle_mod.lm_head_logits(dt.hidden, dt.weight).reshape(B, k + 1, V)
    rng = np.random.default_rng([7, *np.atleast_1d(seed)])
    q = softmax(sharpness * logits[:, :k] + rng.standard_normal((B, k, V)), axis=-1).astype(np.float32)
    temp = temperatures(mode, B)
    tokens = np.empty((B, k), np.int32)
    for b in range(B):
        for i in range(k):
            if temp[b] > 0:
                c = np.cumsum(q[b, i].astype(np.float64))
                tokens[b, i] = min(int(np.searchsorted(c, rng.random() * c[-1], side="right")), V - 1)
            else:
                tokens[b, i] = int(np.argmax(q[b, i]))
    u = rng.random((B, k + 1), dtype=np.float32)
    inp = AcceptInputs(target_logits=logits.astype(np.float32), draft_probs=q, draft_tokens=tokens,
                       uniforms=u, temperature=temp)
    return dt.hidden.reshape(B, k + 1, d), dt.weight, inp, logits


def run_fused(hidden, weight, inp):
    B, k1, d = hidden.shape
    ws = sfv.new_workspace(sfv.verify_lm_head_accept_workspace_size(B, k1 - 1, weight.shape[0]))
    logits, n, toks, ratio = sfv.verify_lm_head_accept(
        bf16_tensor(hidden), bf16_tensor(weight), torch.from_numpy(inp.draft_probs).cuda(),
        torch.from_numpy(inp.draft_tokens).cuda(), torch.from_numpy(inp.uniforms).cuda(),
        torch.from_numpy(inp.temperature).cuda(), workspace=ws)
    torch.cuda.synchronize()
    assert sfv.read_device_status(ws) == 0
    return logits.cpu().numpy(), n.cpu().numpy(), toks.cpu().numpy(), ratio.cpu().numpy()


@pytest.mark.parametrize("B,k,V,d,mode", [
    (1, 5, 32000, 4096, "sampling"),    # image7b acceptance with LLaVA's LM head
    (1, 5, 32000, 4096, "greedy"),
    (8, 6, 6000, 512, "alternate"),
    (4, 8, 3001, 256, "sampling"),      # ragged vocabulary
    (16, 8, 2000, 128, "alternate"),    # 144 rows
    (2, 1, 50, 64, "sampling"),
])
def test_fused_acceptance_matches_oracle(oracle_mod, B, k, V, d, mode):
    hidden, weight, inp, ref_logits = make_case(oracle_mod, B, k, V, d, seed=[B, k, V], mode=mode)
    logits, n, toks, ratio = run_fused(hidden, weight, inp)
    assert np.array_equal(logits.astype(np.float64), ref_logits)
    excluded = compare_accept(oracle_accept(oracle_mod, inp), n, toks, ratio)
    assert excluded <= max(1, B // 10)


def test_fused_agrees_with_unfused_acceptance(oracle_mod):
    hidden, weight, inp, _ = make_case(oracle_mod, 8, 4, 5000, 256, seed=11, mode="alternate",
                                       sharpness=1.5)
    _, n, toks, _ = run_fused(hidden, weight, inp)
    n2, toks2, _ = run_accept(inp)
    assert np.array_equal(n, n2) and np.array_equal(toks, toks2)


def test_fused_qwen_vocabulary(oracle_mod):
    # QwenVL-sized head (152064 x 3584) for 4 sequences with k = 8
    V, d = 152064, HIDDEN_SIZES[152064]
    hidden, weight, inp, ref_logits = make_case(oracle_mod, 4, 8, V, d, seed=5, mode="sampling",
                                                sharpness=1.5)
    logits, n, toks, ratio = run_fused(hidden, weight, inp)
    assert np.array_equal(logits.astype(np.float64), ref_logits)
    compare_accept(oracle_accept(oracle_mod, inp), n, toks, ratio)


def test_fused_invalid_arguments():
    lib = sfv.load_library()
    assert lib.sf_verify_lm_head_accept_workspace_size(32, 8, 1000) == 0  # 288 rows
    assert lib.sf_verify_lm_head_accept_workspace_size(1, 0, 1000) == 0
    assert lib.sf_verify_lm_head_accept_workspace_size(1, 5, 32000) > 0


@pytest.mark.parametrize("V,d", [(152064, 3584), (32000, 4096)])
def test_lm_head_then_accept_on_one_stream(oracle_mod, V, d):
    # The target logits written by sf_lm_head are read by sf_accept launched
    # right after it on the same stream, with no synchronisation between:
    # the projection lets its successor start early, so the acceptance must
    # wait for it before reading any input.  The logits buffer is filled with
    # NaN before each projection, so an early read would show.
    hidden, weight, inp, ref_logits = make_case(oracle_mod, 4, 8, V, d, seed=[21, V], mode="alternate",
                                                sharpness=1.5)
    B, k1, _ = hidden.shape
    h = bf16_tensor(hidden.reshape(B * k1, d))
    w = bf16_tensor(weight)
    dev = {key: torch.from_numpy(getattr(inp, key)).cuda()
           for key in ("draft_probs", "draft_tokens", "uniforms", "temperature")}
    logits = torch.empty((B * k1, V), dtype=torch.float32, device="cuda")
    ws_lm = sfv.new_workspace(sfv.draft_tail_workspace_size(B * k1, V))
    ws_acc = sfv.new_workspace(sfv.accept_workspace_size(B, k1 - 1, V))
    ref = oracle_accept(oracle_mod, inp)
    for _ in range(3):
        logits.fill_(float("nan"))
        sfv.lm_head(h, w, logits=logits, workspace=ws_lm)
        n, toks, ratio = sfv.accept(logits.view(B, k1, V), dev["draft_probs"], dev["draft_tokens"],
                                    dev["uniforms"], dev["temperature"], workspace=ws_acc)
        torch.cuda.synchronize()
        assert np.array_equal(logits.cpu().numpy().reshape(B, k1, V).astype(np.float64), ref_logits)
        assert sfv.read_device_status(ws_acc) == 0
        compare_accept(ref, n.cpu().numpy(), toks.cpu().numpy(), ratio.cpu().numpy())
