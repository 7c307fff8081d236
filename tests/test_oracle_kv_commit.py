"""Pins of the KV-commit oracle (cache bookkeeping after acceptance).

The paper states what happens to the drafts (Sec. 3.1: accepted candidates
join the context, generation continues from the first rejection) but not
how a paged cache is kept; the reading (first min(a + 1, n_q) verified rows
stay, seq_lens prepared for the next n_q_next rows, pages through a free
stack in a fixed order) is written out in the oracle header.  These tests
pin it with hand-worked examples and with invariants any correct bookkeeping
must keep: no page is lost or mapped twice, exactly the needed pages are
mapped, and the kept prefix keeps its physical pages.
"""
import numpy as np
import pytest

from oracle import oracle as om


def commit(seq_lens, block_table, free_pages, free_count, num_accepted, n_q, n_q_next, page=16):
    return om.kv_commit(np.array(seq_lens), np.array(block_table), np.array(free_pages),
                        free_count, np.array(num_accepted), n_q, n_q_next, page)


def test_hand_example_no_page_change():
    # L = 35 - 5 = 30; a = 2 keeps rows 0..2 -> 33 cached; 5 next rows -> 38:
    # pages ceil(35/16) = 3 before, ceil(38/16) = 3 after
    st, sl, bt, fp, fc = commit([35], [[7, 3, 9, -1]], [11, 12, 0, 0], 2, [2], 5, 5)
    assert st == om.ORACLE_OK
    assert sl.tolist() == [38]
    assert bt.tolist() == [[7, 3, 9, -1]]
    assert fc == 2 and fp[:2].tolist() == [11, 12]


def test_hand_example_frees_a_page():
    # 50 tokens on 4 pages; n_q = 10 -> L = 40; a = 0 keeps only row 0 -> 41;
    # 2 next rows -> 43 on 3 pages: logical page 3 (physical 5) is pushed
    st, sl, bt, fp, fc = commit([50], [[4, 8, 1, 5, -1]], [2, 0, 0], 1, [0], 10, 2)
    assert st == om.ORACLE_OK
    assert sl.tolist() == [43]
    assert bt.tolist() == [[4, 8, 1, -1, -1]]
    assert fc == 2 and fp[:2].tolist() == [2, 5]


def test_hand_example_takes_a_page():
    # 32 tokens on 2 pages; n_q = 4 -> L = 28; a = 3 keeps all 4 rows -> 32;
    # 4 next rows -> 36 on 3 pages: the stack top (physical 9) is mapped
    st, sl, bt, fp, fc = commit([32], [[6, 2, -1]], [3, 9], 2, [3], 4, 4)
    assert st == om.ORACLE_OK
    assert sl.tolist() == [36]
    assert bt.tolist() == [[6, 2, 9]]
    assert fc == 1 and fp[0] == 3


def test_hand_example_order_of_pushes_and_takes():
    bt0 = [[10, 11, 20, 30], [40, 41, 42, -1]]
    # n_q = 40, one next row.  seq 0: L = 24, a = 0 keeps 1 -> 25, +1 -> 26 on
    # 2 pages: pushes logical 2 then 3 (physical 20, 30) above [1].  seq 1:
    # L = 0, a = 39 keeps all 40 -> 41 on 3 pages: unchanged.
    st, sl, bt, fp, fc = commit([64, 40], bt0, [1, 0, 0, 0], 1, [0, 39], 40, 1)
    assert st == om.ORACLE_OK
    assert sl.tolist() == [26, 41]
    assert bt.tolist() == [[10, 11, -1, -1], [40, 41, 42, -1]]
    assert fc == 3 and fp[:3].tolist() == [1, 20, 30]
    # nine next rows.  seq 0: 25 + 9 = 34 on 3 pages: pushes 30 -> [1, 30].
    # seq 1: 40 + 9 = 49 on 4 pages: takes the topmost entry, 30.
    st, sl, bt, fp, fc = commit([64, 40], bt0, [1, 0, 0, 0], 1, [0, 39], 40, 9)
    assert st == om.ORACLE_OK
    assert sl.tolist() == [34, 49]
    assert bt.tolist() == [[10, 11, 20, -1], [40, 41, 42, 30]]
    assert fc == 1 and fp[0] == 1
    # 24 next rows.  seq 0: 25 + 24 = 49 on 4 pages: unchanged.  seq 1:
    # 40 + 24 = 64 on 4 pages: takes the stack's only entry, 1.
    st, sl, bt, fp, fc = commit([64, 40], bt0, [1, 0, 0, 0], 1, [0, 39], 40, 24)
    assert st == om.ORACLE_OK
    assert sl.tolist() == [49, 64]
    assert bt.tolist() == [[10, 11, 20, 30], [40, 41, 42, 1]]
    assert fc == 0
    # seq 1 with 33 < n_q tokens is invalid: nothing changes
    st, sl, bt, fp, fc = commit([64, 33], bt0, [1, 0, 0, 0], 1, [0, 8], 40, 1)
    assert st == om.ORACLE_ERR_ARG
    assert bt.tolist() == bt0 and sl.tolist() == [64, 33]


def test_two_taken_pages_are_assigned_bottom_up():
    # stack [5, 6, 7]; one sequence needs two more pages: the two topmost
    # entries, the lower one (6) for the lower logical page
    st, sl, bt, fp, fc = commit([16], [[9, -1, -1]], [5, 6, 7], 3, [3], 4, 20)
    # L = 12, keep 4 -> 16, next 20 -> 36 on 3 pages
    assert st == om.ORACLE_OK
    assert bt.tolist() == [[9, 6, 7]]
    assert fc == 1 and fp[0] == 5


def test_out_of_pages_and_overflow_change_nothing():
    args = ([16], [[9, -1, -1]], [5, 0, 0], 1, [3], 4, 20)
    st, sl, bt, fp, fc = commit(*args)
    assert st == om.ORACLE_ERR_PAGES
    assert sl.tolist() == [16] and bt.tolist() == [[9, -1, -1]] and fc == 1
    # pushes beyond the stack capacity
    st, sl, bt, fp, fc = commit([48], [[1, 2, 3]], [7], 1, [0], 32, 1)
    assert st == om.ORACLE_ERR_PAGES and bt.tolist() == [[1, 2, 3]]


def test_invalid_sequences_change_nothing():
    assert commit([3], [[1]], [0], 0, [0], 4, 1)[0] == om.ORACLE_ERR_ARG       # seq_len < n_q
    assert commit([16], [[1]], [0], 0, [-1], 4, 1)[0] == om.ORACLE_ERR_ARG     # a < 0
    assert commit([16], [[1]], [2, 3], 2, [3], 4, 4)[0] == om.ORACLE_ERR_ARG   # needs 2 > 1 pages


def random_state(rng, B, max_pages, n_q, pool_extra=8):
    lens = rng.integers(n_q, max_pages * 16 - 40, size=B)
    had = (lens + 15) // 16
    pool = rng.permutation(int(had.sum()) + pool_extra + int(B * 3))
    bt = np.full((B, max_pages), -1, np.int64)
    pos = 0
    for b in range(B):
        bt[b, :had[b]] = pool[pos:pos + had[b]]
        pos += had[b]
    free = pool[pos:]
    cap = len(free) + int(had.sum())
    fp = np.zeros(cap, np.int64)
    fp[:len(free)] = free
    return lens, bt, fp, len(free)


@pytest.mark.parametrize("seed", range(40))
def test_invariants_on_random_batches(seed):
    rng = np.random.default_rng(seed)
    B, max_pages = int(rng.integers(1, 40)), int(rng.integers(6, 40))
    n_q, n_q_next = int(rng.integers(1, 17)), int(rng.integers(1, 17))
    lens, bt, fp, fc = random_state(rng, B, max_pages, n_q)
    acc = rng.integers(0, 18, size=B)
    st, sl2, bt2, fp2, fc2 = commit(lens, bt, fp, fc, acc, n_q, n_q_next)
    assert st == om.ORACLE_OK
    # at least one verified row (the block's first token) always stays, and
    # never more than the n_q verified ones
    assert np.all(sl2 >= lens - n_q + 1 + n_q_next)
    assert np.all(sl2 <= lens + n_q_next)
    # conservation: the multiset of pages is unchanged
    before = sorted([int(x) for b in range(B) for x in bt[b, :(lens[b] + 15) // 16]] +
                    [int(x) for x in fp[:fc]])
    after = sorted([int(x) for x in bt2[bt2 >= 0]] + [int(x) for x in fp2[:fc2]])
    assert before == after
    for b in range(B):
        need = (int(sl2[b]) + 15) // 16
        # coverage: exactly the needed logical pages are mapped
        assert np.all(bt2[b, :need] >= 0) and np.all(bt2[b, need:] == -1)
        # the kept prefix stays on its physical pages
        common = min(need, (int(lens[b]) + 15) // 16)
        assert np.array_equal(bt2[b, :common], bt[b, :common])


def test_accepting_more_keeps_more_until_all_rows_are_kept():
    rng = np.random.default_rng(7)
    lens, bt, fp, fc = random_state(rng, 1, 20, 6)
    prev = None
    for a in range(0, 9):
        st, sl2, *_ = commit(lens, bt, fp, fc, [a], 6, 3)
        assert st == om.ORACLE_OK
        if prev is not None:
            assert sl2[0] == prev + (1 if a < 6 else 0)
        prev = int(sl2[0])
    assert prev == lens[0] + 3
