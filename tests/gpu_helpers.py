"""Shared helpers of the GPU parity tests: move seeded numpy inputs to the
device, run the CUDA path through the C ABI, and compare with the oracle."""
import numpy as np
import pytest
import torch

from paper_2505_12728_gb300 import build_lib
from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import bf16_bits_to_f32

# Tolerances of the verification attention against the fp64 oracle for bf16
# inputs: max abs error of the bf16 output and of the fp32 LSE.
ATTN_OUT_ATOL = 1e-2
ATTN_LSE_ATOL = 1e-3
# Decisions whose oracle margin is below this are excluded from bit-exact
# comparison (a CDF boundary or acceptance threshold within 1e-6 of u).
MARGIN = 1e-6


def require_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build_lib.build()
    sfv.load_library()


def bf16_tensor(bits: np.ndarray, device="cuda"):
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


def attention_to_device(case, layer=0):
    return dict(q=bf16_tensor(case.q[layer]), k_cache=bf16_tensor(case.k_cache[layer]),
                v_cache=bf16_tensor(case.v_cache[layer]),
                block_table=torch.from_numpy(case.block_table[layer]).cuda(),
                seq_lens=torch.from_numpy(case.seq_lens).cuda())


def run_attention(case, layer=0, num_splits=0, workspace=None, dev=None):
    dev = dev or attention_to_device(case, layer)
    out, lse = sfv.verify_attention(dev["q"], dev["k_cache"], dev["v_cache"], dev["block_table"],
                                    dev["seq_lens"], num_splits=num_splits, workspace=workspace)
    torch.cuda.synchronize()
    return out.float().cpu().numpy(), lse.cpu().numpy()


def oracle_attention(oracle_mod, case, layer=0, select=(-1, -1, -1)):
    return oracle_mod.verify_attention(case.q[layer], case.k_cache[layer], case.v_cache[layer],
                                       case.block_table[layer], case.seq_lens, H_kv=case.H_kv,
                                       select=select)


def bf16_half_ulp(x):
    """Half the spacing of bf16 values at |x| (8 significant bits): the
    error of rounding the exact value to the bf16 output format."""
    a = np.abs(np.asarray(x, np.float64))
    a = np.where(np.isfinite(a), a, 0.0)  # (unselected oracle entries are NaN)
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return np.ldexp(1.0, e.astype(np.int64) - 8)


def assert_attention_close(out, lse, ref_out, ref_lse, mask=None):
    """Max abs error ATTN_OUT_ATOL on the output beyond its own bf16 rounding
    (half a bf16 ulp of the exact value: 2^-6 at |o| in [4, 8), more than the
    bound itself), and ATTN_LSE_ATOL on the fp32 LSE."""
    if mask is None:
        mask = np.ones(ref_lse.shape, bool)
    err_o = (np.abs(out - ref_out) - bf16_half_ulp(ref_out))[mask].max()
    err_l = np.abs(lse - ref_lse)[mask].max()
    assert np.isfinite(out[mask]).all() and np.isfinite(lse[mask]).all()
    assert err_o <= ATTN_OUT_ATOL, f"max |out - oracle| = {err_o}"
    assert err_l <= ATTN_LSE_ATOL, f"max |lse - oracle| = {err_l}"
    return err_o, err_l


def accept_to_device(inp):
    return dict(target_logits=torch.from_numpy(inp.target_logits).cuda(),
                draft_probs=torch.from_numpy(inp.draft_probs).cuda(),
                draft_tokens=torch.from_numpy(inp.draft_tokens).cuda(),
                uniforms=torch.from_numpy(inp.uniforms).cuda(),
                temperature=torch.from_numpy(inp.temperature).cuda())


def run_accept(inp, workspace=None, dev=None):
    dev = dev or accept_to_device(inp)
    n, toks, ratio = sfv.accept(dev["target_logits"], dev["draft_probs"], dev["draft_tokens"],
                                dev["uniforms"], dev["temperature"], workspace=workspace)
    torch.cuda.synchronize()
    return n.cpu().numpy(), toks.cpu().numpy(), ratio.cpu().numpy()


def oracle_accept(oracle_mod, inp):
    return oracle_mod.accept(inp.target_logits, inp.draft_probs, inp.draft_tokens, inp.uniforms,
                             inp.temperature)


def compare_accept(ref, n, toks, ratio, ratio_atol=2e-6):
    """Bit-exact accepted lengths and tokens for every sequence whose oracle
    decisions all have a margin >= MARGIN; returns the number excluded."""
    B = n.shape[0]
    excluded = 0
    for b in range(B):
        j = int(ref["num_accepted"][b])
        k = ref["margin"].shape[1] - 1
        decided = list(range(min(j + 1, k))) + [k]
        if (ref["margin"][b, decided] < MARGIN).any():
            excluded += 1
            continue
        assert int(n[b]) == j, (b, int(n[b]), j)
        np.testing.assert_array_equal(toks[b], ref["out_tokens"][b], err_msg=f"sequence {b}")
    np.testing.assert_allclose(ratio, ref["accept_ratio"], rtol=0, atol=ratio_atol)
    return excluded


def bits_to_float(bits):
    return bf16_bits_to_f32(bits)
