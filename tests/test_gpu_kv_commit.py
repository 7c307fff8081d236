"""GPU parity of sf_kv_commit against the oracle (bit-exact), and a decoding
loop that closes the verification step: verify -> accept -> commit -> append
the next draft rows' K/V -> verify, checked against the oracle every round."""
import numpy as np
import pytest
import torch

from paper_2505_12728_gb300 import specflash_verify as sfv
from paper_2505_12728_gb300.workloads import f32_to_bf16_bits, make_attention_case
from tests.gpu_helpers import assert_attention_close, require_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def random_state(rng, B, max_pages, n_q, spare):
    lens = rng.integers(n_q, max_pages * 16 - 40, size=B).astype(np.int32)
    had = (lens + 15) // 16
    pool = rng.permutation(int(had.sum()) + spare).astype(np.int32)
    bt = np.full((B, max_pages), -1, np.int32)
    pos = 0
    for b in range(B):
        bt[b, :had[b]] = pool[pos:pos + had[b]]
        pos += had[b]
    free = pool[pos:]
    fp = np.zeros(len(free) + int(had.sum()), np.int32)
    fp[:len(free)] = free
    return lens, bt, fp, len(free)


def gpu_commit(lens, bt, fp, fc, acc, n_q, n_q_next):
    t = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (lens, bt, fp)]
    tfc = torch.tensor([fc], dtype=torch.int32, device="cuda")
    tacc = torch.from_numpy(np.ascontiguousarray(acc, dtype=np.int32)).cuda()
    ws = sfv.new_workspace(sfv.kv_commit_workspace_size())
    sfv.kv_commit(t[0], t[1], t[2], tfc, tacc, n_q, n_q_next, workspace=ws)
    torch.cuda.synchronize()
    return (sfv.read_device_status(ws), t[0].cpu().numpy(), t[1].cpu().numpy(),
            t[2].cpu().numpy(), int(tfc.item()))


@pytest.mark.parametrize("seed", range(12))
def test_random_batches_match_oracle(oracle_mod, seed):
    rng = np.random.default_rng(100 + seed)
    B = int(rng.choice([1, 7, 64, 333, 1024]))
    max_pages = int(rng.integers(4, 60))
    n_q, n_q_next = int(rng.integers(1, 17)), int(rng.integers(1, 17))
    lens, bt, fp, fc = random_state(rng, B, max_pages, n_q, spare=4 * B)
    acc = rng.integers(0, 17, size=B).astype(np.int32)
    st, sl, bt2, fp2, fc2 = gpu_commit(lens, bt, fp, fc, acc, n_q, n_q_next)
    ost, osl, obt, ofp, ofc = oracle_mod.kv_commit(lens, bt, fp, fc, acc, n_q, n_q_next)
    assert ost == oracle_mod.ORACLE_OK and st == 0
    np.testing.assert_array_equal(sl, osl)
    np.testing.assert_array_equal(bt2, obt)
    np.testing.assert_array_equal(fp2, ofp)
    assert fc2 == ofc


def test_page_shortage_sets_status_and_changes_nothing(oracle_mod):
    lens = np.array([16, 30], np.int32)
    bt = np.array([[9, -1, -1], [4, 5, -1]], np.int32)
    fp = np.array([7, 0, 0], np.int32)
    acc = np.array([3, 3], np.int32)
    st, sl, bt2, fp2, fc2 = gpu_commit(lens, bt, fp, 1, acc, 4, 16)
    assert oracle_mod.kv_commit(lens, bt, fp, 1, acc, 4, 16)[0] == oracle_mod.ORACLE_ERR_PAGES
    assert st & sfv.SF_DEVICE_OUT_OF_PAGES
    np.testing.assert_array_equal(sl, lens)
    np.testing.assert_array_equal(bt2, bt)
    np.testing.assert_array_equal(fp2, fp)
    assert fc2 == 1


def test_invalid_sequence_sets_status_and_changes_nothing():
    lens = np.array([16, 3], np.int32)       # 3 < n_q
    bt = np.array([[9, -1], [4, -1]], np.int32)
    fp = np.array([7, 8], np.int32)
    st, sl, bt2, fp2, fc2 = gpu_commit(lens, bt, fp, 2, np.array([0, 0], np.int32), 4, 4)
    assert st & sfv.SF_DEVICE_BAD_SEQLEN
    np.testing.assert_array_equal(sl, lens)
    np.testing.assert_array_equal(bt2, bt)
    assert fc2 == 2


def test_invalid_arguments_raise_before_launch():
    z = torch.zeros(4, dtype=torch.int32, device="cuda")
    bt = torch.zeros((4, 8), dtype=torch.int32, device="cuda")
    fc = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(sfv.SFError):
        sfv.kv_commit(z, bt, z, fc, z, 0, 4)          # n_q = 0
    with pytest.raises(sfv.SFError):
        sfv.kv_commit(z, bt, z, fc, z, 4, 17)         # n_q_next > 16
    with pytest.raises(sfv.SFError):
        sfv.kv_commit(z, bt, z, fc, z, 4, 4, workspace=sfv.new_workspace(64))


def test_three_round_decoding_loop_matches_oracle(oracle_mod):
    # B = 3 sequences, 8/2 heads, d = 128, k = 4 drafts, n_q = k + 1 rows per
    # step, vocabulary 64.  Each round: append the n_q new rows' K/V at the
    # committed length, verify, accept, commit -- on the GPU and with the
    # oracle, comparing attention (tolerance) and everything else (exactly).
    rng = np.random.default_rng(5)
    B, H_q, H_kv, d, k, V = 3, 8, 2, 128, 4, 64
    n_q = k + 1
    case = make_attention_case(B, n_q, H_q, H_kv, d, [100, 37, 250], seed=321, spare_pages=40)
    kc, vc = case.k_cache[0].copy(), case.v_cache[0].copy()
    # room for the sequences to grow by up to n_q tokens per round
    num_pages, max_pages = kc.shape[0], case.block_table.shape[2] + 4
    lens = case.seq_lens.astype(np.int32).copy()
    bt = np.full((B, max_pages), -1, np.int32)
    bt[:, :case.block_table.shape[2]] = case.block_table[0]
    used = set(int(x) for b in range(B) for x in bt[b, :(lens[b] + 15) // 16])
    free = np.array([p for p in range(num_pages) if p not in used], np.int32)
    fp = np.zeros(num_pages, np.int32)
    fp[:len(free)] = free
    fc = len(free)
    d_kc = torch.from_numpy(kc.view(np.int16)).cuda().view(torch.bfloat16)
    d_vc = torch.from_numpy(vc.view(np.int16)).cuda().view(torch.bfloat16)
    d_lens, d_bt = torch.from_numpy(lens).cuda(), torch.from_numpy(bt).cuda()
    d_fp, d_fc = torch.from_numpy(fp).cuda(), torch.tensor([fc], dtype=torch.int32, device="cuda")
    ws_att = sfv.new_workspace(sfv.verify_attention_workspace_size(B, n_q, H_q, H_kv, d, max_pages))
    ws_acc = sfv.new_workspace(sfv.accept_workspace_size(B, k, V))
    ws_com = sfv.new_workspace(sfv.kv_commit_workspace_size())
    for rnd in range(3):
        # the new rows' K/V at positions L_b .. L_b + n_q - 1 (the "append")
        q = f32_to_bf16_bits(rng.standard_normal((B, n_q, H_q, d)).astype(np.float32))
        for b in range(B):
            L = int(lens[b]) - n_q
            for i in range(n_q):
                pos = L + i
                page, slot = int(bt[b, pos // 16]), pos % 16
                kc[page, :, slot, :] = f32_to_bf16_bits(rng.standard_normal((H_kv, d)).astype(np.float32))
                vc[page, :, slot, :] = f32_to_bf16_bits(rng.standard_normal((H_kv, d)).astype(np.float32))
        d_kc.copy_(torch.from_numpy(kc.view(np.int16)).cuda().view(torch.bfloat16))
        d_vc.copy_(torch.from_numpy(vc.view(np.int16)).cuda().view(torch.bfloat16))
        d_q = torch.from_numpy(q.view(np.int16)).cuda().view(torch.bfloat16)
        out, lse = sfv.verify_attention(d_q, d_kc, d_vc, d_bt, d_lens, workspace=ws_att)
        ref_out, ref_lse = oracle_mod.verify_attention(q, kc, vc, bt, lens, H_kv=H_kv)
        torch.cuda.synchronize()
        assert_attention_close(out.float().cpu().numpy(), lse.cpu().numpy(), ref_out, ref_lse)
        # acceptance on small synthetic distributions
        logits = (rng.standard_normal((B, k + 1, V)) * 3).astype(np.float32)
        qp = np.exp(logits[:, :k] + rng.standard_normal((B, k, V)).astype(np.float32))
        qp = (qp / qp.sum(-1, keepdims=True)).astype(np.float32)
        toks = np.array([[rng.choice(V, p=qp[b, i] / qp[b, i].sum()) for i in range(k)]
                         for b in range(B)], np.int32)
        uni = rng.random((B, k + 1)).astype(np.float32)
        tau = np.ones(B, np.float32)
        g = [torch.from_numpy(x).cuda() for x in (logits, qp, toks, uni, tau)]
        n_acc, out_tok, _ = sfv.accept(*g, workspace=ws_acc)
        ref_acc = oracle_mod.accept(logits, qp, toks, uni, tau)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(n_acc.cpu().numpy(), ref_acc["num_accepted"])
        # commit on the GPU, and the same with the oracle on host copies
        sfv.kv_commit(d_lens, d_bt, d_fp, d_fc, n_acc, n_q, n_q, workspace=ws_com)
        ost, lens, bt, fp, fc = oracle_mod.kv_commit(lens, bt, fp, fc, ref_acc["num_accepted"],
                                                     n_q, n_q)
        torch.cuda.synchronize()
        assert ost == oracle_mod.ORACLE_OK
        np.testing.assert_array_equal(d_lens.cpu().numpy(), lens)
        np.testing.assert_array_equal(d_bt.cpu().numpy(), bt)
        np.testing.assert_array_equal(d_fp.cpu().numpy(), fp)
        assert int(d_fc.item()) == fc
    assert sfv.read_device_status(ws_att) == 0 and sfv.read_device_status(ws_com) == 0
