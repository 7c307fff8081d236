"""GPU parity of sf_verify_attention against the fp64 oracle (C ABI path).

Tolerances (bf16 inputs, fp32 accumulation): max abs error 1e-2 on the bf16
output beyond its own rounding to bf16 (half a bf16 ulp of the exact value),
and 1e-3 on the LSE, at every output element compared.
"""
import math

import numpy as np
import pytest
import torch

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import (WORKLOADS, f32_to_bf16_bits, make_attention_case,
                                              make_attention_inputs, workload)
from tests.gpu_helpers import (assert_attention_close, attention_to_device, oracle_attention,
                               require_gpu, run_attention)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


EDGE_CASES = [
    # (B, n_q, H_q, H_kv, d, prefixes)
    (1, 1, 8, 8, 64, [0]),
    (1, 1, 8, 8, 128, [1]),
    (2, 4, 8, 8, 64, [15, 16]),
    (2, 5, 32, 32, 128, [17, 63]),
    (3, 8, 28, 4, 128, [64, 65, 200]),
    (2, 16, 8, 1, 64, [0, 47]),
    (2, 16, 16, 2, 128, [300, 1]),
    (1, 6, 7, 1, 128, [129]),
    (4, 2, 12, 3, 64, [5, 70, 133, 16]),
    (2, 9, 28, 4, 128, [1000, 777]),
    (1, 3, 16, 2, 128, [0]),
]


@pytest.mark.parametrize("case_idx", range(len(EDGE_CASES)))
@pytest.mark.parametrize("num_splits", [0, 1, 2, 7])
def test_edge_shapes_match_oracle(oracle_mod, case_idx, num_splits):
    B, n_q, H_q, H_kv, d, prefixes = EDGE_CASES[case_idx]
    case = make_attention_case(B, n_q, H_q, H_kv, d, prefixes, seed=1000 + case_idx,
                               spare_pages=3)
    out, lse = run_attention(case, num_splits=num_splits)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    assert_attention_close(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("name", ["tiny", "gqa", "video"])
def test_named_workloads_match_oracle(oracle_mod, name):
    wl = WORKLOADS[name]
    case = make_attention_inputs(wl)
    out, lse = run_attention(case)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    assert_attention_close(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("n_q_extra", [0, 1])
def test_image7b_all_layers_match_oracle(oracle_mod, n_q_extra):
    # 32 independent layers (separate caches), n_q = k and n_q = k + 1.
    wl = workload("image7b", n_q=WORKLOADS["image7b"].k + n_q_extra)
    case = make_attention_inputs(wl)
    for layer in range(case.layers):
        out, lse = run_attention(case, layer=layer)
        ref_out, ref_lse = oracle_attention(oracle_mod, case, layer=layer)
        assert_attention_close(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("k", [2, 4, 8])
def test_long_video_sampled_rows_match_oracle(oracle_mod, k):
    # Full-size long-context workload (B=16, prefixes up to 32768 tokens) in
    # the launch configuration the benchmark uses; the oracle computes 48
    # sampled (sequence, row, head) outputs one by one.
    wl = workload("long", k=k)
    case = make_attention_inputs(wl)
    out, lse = run_attention(case)
    rng = np.random.default_rng(k)
    picks = {(int(rng.integers(wl.B)), int(rng.integers(wl.rows)), int(rng.integers(wl.H_q)))
             for _ in range(48)}
    picks |= {(wl.B - 1, wl.rows - 1, wl.H_q - 1), (0, 0, 0)}
    for b, i, h in sorted(picks):
        ref_out, ref_lse = oracle_attention(oracle_mod, case, select=(b, i, h))
        mask = np.zeros(ref_lse.shape, bool)
        mask[b, i, h] = True
        assert_attention_close(out, lse, ref_out, ref_lse, mask=mask)


def test_split_count_changes_only_rounding(oracle_mod):
    case = make_attention_case(4, 8, 28, 4, 128, [900, 2000, 64, 1500], seed=77)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    outs = []
    for splits in (1, 3, 16, 100, 0):
        out, lse = run_attention(case, num_splits=splits)
        assert_attention_close(out, lse, ref_out, ref_lse)
        outs.append(out)
    for o in outs[1:]:
        assert np.abs(o - outs[0]).max() <= 2e-2


def test_repeated_calls_are_bit_identical():
    case = make_attention_case(3, 6, 28, 4, 128, [700, 1900, 33], seed=78)
    dev = attention_to_device(case)
    ws = sfv.new_workspace(sfv.verify_attention_workspace_size(3, 6, 28, 4, 128,
                                                               case.block_table.shape[2]))
    a = run_attention(case, dev=dev, workspace=ws)
    b = run_attention(case, dev=dev, workspace=ws)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])
    assert sfv.read_device_status(ws) == 0


def test_garbage_past_sequence_end_is_ignored(oracle_mod):
    # Slots past seq_len in the last page hold NaN/Inf: outputs stay exact.
    case = make_attention_case(2, 5, 8, 2, 128, [21, 90], seed=79)
    kc, vc = case.k_cache.copy(), case.v_cache.copy()
    nan = f32_to_bf16_bits(np.array([np.nan], np.float32))[0]
    inf = f32_to_bf16_bits(np.array([np.inf], np.float32))[0]
    for b in range(2):
        T = int(case.seq_lens[b])
        last = case.block_table[0, b, (T - 1) // 16]
        kc[0, last, :, T % 16:, :] = inf
        vc[0, last, :, T % 16:, :] = nan
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    case.k_cache, case.v_cache = kc, vc
    out, lse = run_attention(case)
    assert_attention_close(out, lse, ref_out, ref_lse)


def test_out_of_range_page_sets_status_without_fault(oracle_mod):
    case = make_attention_case(2, 4, 8, 2, 64, [100, 60], seed=80)
    bt = case.block_table.copy()
    bt[0, 1, 2] = case.k_cache.shape[1] + 5          # sequence 1, logical page 2
    dev = attention_to_device(case)
    dev["block_table"] = torch.from_numpy(bt[0]).cuda()
    ws = sfv.new_workspace(sfv.verify_attention_workspace_size(2, 4, 8, 2, 64, bt.shape[2]))
    out, lse = run_attention(case, dev=dev, workspace=ws)
    assert sfv.read_device_status(ws) & sfv.SF_DEVICE_BAD_PAGE
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    mask = np.zeros(ref_lse.shape, bool)
    mask[0] = True                                     # sequence 0 is untouched
    assert_attention_close(out, lse, ref_out, ref_lse, mask=mask)
    assert np.isfinite(out).all()


def test_bad_seq_len_is_flagged_and_clamped():
    case = make_attention_case(2, 4, 8, 2, 64, [30, 30], seed=81)
    dev = attention_to_device(case)
    dev["seq_lens"] = torch.tensor([2, 10 ** 6], dtype=torch.int32, device="cuda")
    ws = sfv.new_workspace(sfv.verify_attention_workspace_size(2, 4, 8, 2, 64,
                                                               case.block_table.shape[2]))
    out, lse = run_attention(case, dev=dev, workspace=ws)
    assert sfv.read_device_status(ws) & sfv.SF_DEVICE_BAD_SEQLEN
    assert np.isfinite(out).all() and np.isfinite(lse).all()


def test_explicit_softmax_scale(oracle_mod):
    case = make_attention_case(1, 4, 8, 8, 64, [50], seed=82)
    dev = attention_to_device(case)
    out, lse = sfv.verify_attention(dev["q"], dev["k_cache"], dev["v_cache"], dev["block_table"],
                                    dev["seq_lens"], softmax_scale=0.05)
    ref_out, ref_lse = oracle_mod.verify_attention(case.q[0], case.k_cache[0], case.v_cache[0],
                                                   case.block_table[0], case.seq_lens, H_kv=8,
                                                   scale=0.05)
    assert_attention_close(out.float().cpu().numpy(), lse.cpu().numpy(), ref_out, ref_lse)


def test_invalid_arguments_raise_before_launch():
    case = make_attention_case(1, 4, 8, 8, 64, [10], seed=83)
    dev = attention_to_device(case)
    with pytest.raises(sfv.SFError):      # 7 query heads over 2 KV heads
        sfv.verify_attention(dev["q"][:, :, :7].contiguous(), dev["k_cache"][:, :2].contiguous(),
                             dev["v_cache"][:, :2].contiguous(), dev["block_table"],
                             dev["seq_lens"])
    with pytest.raises(sfv.SFError):      # workspace too small
        sfv.verify_attention(dev["q"], dev["k_cache"], dev["v_cache"], dev["block_table"],
                             dev["seq_lens"], workspace=sfv.new_workspace(256))


@pytest.mark.parametrize("B,n_q,H_q,H_kv,d,prefix", [
    (1, 5, 32, 32, 128, 3008),     # one sequence, MHA: one 8-CTA cluster per KV head
    (1, 8, 128, 32, 128, 2000),    # one sequence, 32 rows per KV head
    (1, 7, 224, 32, 64, 700),      # one sequence, 49 rows per KV head, d = 64
    (2, 8, 28, 4, 128, 2000),      # equal-length batch (balanced global partition)
])
def test_uniform_segments_match_oracle(oracle_mod, B, n_q, H_q, H_kv, d, prefix):
    # With the automatic split count a single sequence's segments are each
    # covered by one thread-block cluster whose CTAs merge through
    # distributed shared memory; results must match the oracle like every
    # other path, and repeat bit for bit.
    case = make_attention_case(B, n_q, H_q, H_kv, d, [prefix] * B, seed=900 + B + n_q)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    out, lse = run_attention(case, num_splits=0)
    assert_attention_close(out, lse, ref_out, ref_lse)
    out2, lse2 = run_attention(case, num_splits=0)
    np.testing.assert_array_equal(out, out2)


@pytest.mark.parametrize("n_q,H_q,H_kv", [(8, 28, 4), (3, 16, 2), (1, 8, 8)])
def test_growing_scores_move_the_running_maximum(oracle_mod, n_q, H_q, H_kv):
    # Scores that grow along the sequence (q all ones, every element of key t
    # equal to t / 64) raise each row's maximum by about 16 (base 2) per
    # 64-key tile, far beyond any lazy-rescale threshold, so the running
    # output and sum are rescaled at every tile of every piece.
    case = make_attention_case(2, n_q, H_q, H_kv, 128, [900, 1500], seed=95, spare_pages=2)
    one = f32_to_bf16_bits(np.array([1.0], np.float32))[0]
    case.q[...] = one
    for b in range(2):
        for t in range(int(case.seq_lens[b])):
            page = case.block_table[0, b, t // 16]
            case.k_cache[0, page, :, t % 16, :] = f32_to_bf16_bits(np.array([t / 64.0], np.float32))[0]
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    for splits in (0, 3):
        out, lse = run_attention(case, num_splits=splits)
        assert_attention_close(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("prefix,max_pages", [
    (1200, None),   # 76 pages, row of 76 entries: copied to shared memory
    (1200, 512),    # row of 512 entries (436 unused, -1): copied
    (1200, 513),    # one entry wider: read from global memory
    (8187, None),   # 8192 tokens = 512 pages, every entry used: copied
    (8188, None),   # 513 pages: read from global memory
])
def test_one_sequence_block_table_row_widths(oracle_mod, prefix, max_pages):
    # A single sequence's block-table row of up to 512 entries is copied to
    # shared memory at kernel entry; wider rows are read from global memory.
    # Both sides of that limit, with and without unused entries, must give
    # the oracle's result on the 8-CTA cluster path.
    case = make_attention_case(1, 5, 32, 32, 128, [prefix], seed=1300 + prefix % 97,
                               max_pages=max_pages)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    out, lse = run_attention(case, num_splits=0)
    assert_attention_close(out, lse, ref_out, ref_lse)


def test_kernel_launch_counts_follow_the_rows_per_kv_head():
    # at most 16 rows per KV head: one launch (the split kernel merges in
    # place); more: the tcgen05 split kernel and its merge kernel
    assert sfv.verify_attention_kernel_launches(1, 5, 32, 32, 128, 189) == 1
    assert sfv.verify_attention_kernel_launches(2, 16, 8, 8, 64, 40) == 1
    assert sfv.verify_attention_kernel_launches(4, 8, 28, 4, 128, 305) == 2
    assert sfv.verify_attention_kernel_launches(16, 8, 28, 4, 128, 2049) == 2


@pytest.mark.parametrize("B,n_q,H_q,H_kv,d,prefix_range", [
    (1, 16, 8, 1, 128, (20000, 20000)),  # one 128-row segment over every CTA
    (1, 16, 8, 1, 64, (20000, 20000)),
    (1, 8, 28, 4, 128, (30000, 30000)),  # four 56-row segments of ~38 pieces each
    (1, 4, 28, 4, 128, (30000, 30000)),  # 28 rows (four key-split copies): ~152
                                         # partials per segment and row
    (2, 3, 16, 2, 64, (12000, 12000)),   # 24 rows, head_dim 64, four copies
    (40, 8, 28, 4, 128, (500, 3000)),    # 160 segments > 152 CTAs: balanced partition,
                                         # a CTA's first and last pieces split
])
def test_tcgen05_many_piece_merges_match_oracle(oracle_mod, B, n_q, H_q, H_kv, d, prefix_range):
    # Segments split over many CTAs (up to every CTA of the grid, 128 rows)
    # and CTAs holding pieces of several segments: the merge kernel combines
    # the partials of all pieces of each split segment, in batches.
    rng = np.random.default_rng(4000 + B + d)
    prefixes = [int(x) for x in rng.integers(prefix_range[0], prefix_range[1] + 1, size=B)]
    case = make_attention_case(B, n_q, H_q, H_kv, d, prefixes, seed=4100 + B + d)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    for splits in (0, 37):
        out, lse = run_attention(case, num_splits=splits)
        assert_attention_close(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("n_q,H_q,H_kv,d", [
    (4, 8, 8, 64),      # mma.sync kernel: 8192 segments of one or two tiles
    (8, 28, 4, 128),    # tcgen05 kernel: 56 rows per KV head, 4096 segments
])
def test_largest_batch_matches_oracle(oracle_mod, n_q, H_q, H_kv, d):
    # B = 1024 sequences (the batch limit) with ragged prefixes of 0..120
    # tokens: the on-device tile partition spans every sequence
    rng = np.random.default_rng(1024 + n_q)
    prefixes = [int(x) for x in rng.integers(0, 121, size=1024)]
    case = make_attention_case(1024, n_q, H_q, H_kv, d, prefixes, seed=77 + d)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    out, lse = run_attention(case, num_splits=0)
    assert_attention_close(out, lse, ref_out, ref_lse)


def test_outputs_beyond_four_are_judged_against_their_bf16_rounding(oracle_mod):
    # Rows with two visible keys give outputs near single V entries, up to
    # ~4.4 here.  bf16 values in [4, 8) are 2^-5 apart: the exact -4.3895 can
    # only be written as -4.375, 0.0145 away, more than the 1e-2 bound.  The
    # kernel writes the correctly rounded value; the bound applies beyond it.
    prefixes = [4112, 129, 17, 15, 64, 0, 15, 1, 4329, 3479, 63, 124, 183, 3530, 2894, 0]
    case = make_attention_case(16, 10, 32, 8, 128, prefixes, seed=200206, spare_pages=3)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    out, lse = run_attention(case, num_splits=7)
    assert np.abs(out - ref_out).max() > 1e-2           # the bf16 format alone
    assert_attention_close(out, lse, ref_out, ref_lse)  # within 1e-2 beyond it


def test_a_wait_that_runs_out_reports_a_timeout_and_the_context_stays_usable(oracle_mod):
    # The bounded wait the kernels use, on an mbarrier nothing completes:
    # after ~1 s it gives up and sets SF_DEVICE_TIMEOUT; no fault, no hang.
    import time
    ws = sfv.new_workspace(256)
    t0 = time.time()
    sfv.selftest_bounded_wait(ws)
    assert sfv.read_device_status(ws) == sfv.SF_DEVICE_TIMEOUT
    assert 0.5 < time.time() - t0 < 30
    # the context still runs both kernels correctly
    case = make_attention_case(2, 8, 28, 4, 128, [300, 1000], seed=85)
    out, lse = run_attention(case)
    ref_out, ref_lse = oracle_attention(oracle_mod, case)
    assert_attention_close(out, lse, ref_out, ref_lse)
