"""Pins of the plain-Python KV bookkeeping model (oracle/kv.py) on the CPU: hand-worked cases and the
invariants of the pool (every page exactly once: in a table or on the free stack)."""
import numpy as np

from oracle import kv


def _fresh(num_blocks, B, max_blocks):
    return [[-1] * max_blocks for _ in range(B)], list(range(num_blocks)), num_blocks


def test_hand_worked_reserve_and_commit():
    tables, stack, F = _fresh(8, 2, 4)
    # request 0: c=20, k=3 -> tokens 0..23 -> 2 pages; request 1: c=0, k=0 -> 1 page
    F, codes = kv.reserve_append(tables, stack, F, [20, 0], [3, 0], 8)
    assert codes == [0, 0] and F == 5
    assert tables[0][:2] == [7, 6] and tables[1][:1] == [5]   # popped from the top, table order
    ctx = [20, 0]
    # request 0 accepts 0 of 3: c' = 21 -> still 2 pages; request 1 accepts 0 of 0: c' = 1
    F, codes = kv.commit(tables, stack, F, ctx, [3, 0], [0, 0])
    assert codes == [0, 0] and ctx == [21, 1] and F == 5
    # request 0 with c=10, k=9 (tokens 0..19, 2 pages) rejects everything: c' = 11 -> page 1 freed
    t2, s2, F2 = [[3, 4, -1, -1]], [0, 1, 2, 5, 6, 7, -1, -1], 6
    F2, codes = kv.commit(t2, s2, F2, [10], [9], [0])
    assert codes == [0] and t2[0] == [3, -1, -1, -1] and F2 == 7 and s2[6] == 4


def test_exhaustion_serves_a_prefix_and_flags_the_rest():
    tables, stack, F = _fresh(3, 3, 4)
    F, codes = kv.reserve_append(tables, stack, F, [0, 30, 0], [0, 1, 0], 3)   # needs 1, 2, 1 pages
    assert codes == [0, 0, kv.NO_BLOCKS] and F == 0 and tables[2] == [-1] * 4


def test_bad_lengths_are_flagged_and_skipped():
    tables, stack, F = _fresh(4, 2, 2)
    F, codes = kv.reserve_append(tables, stack, F, [40, 0], [0, -1], 4)   # 41 tokens > 32; k < 0
    assert codes == [kv.BAD_LENGTH, kv.BAD_LENGTH] and F == 4
    F, codes = kv.commit(tables, stack, F, [0, 0], [2, 2], [3, -1])       # L > k; L < 0
    assert codes == [kv.BAD_LENGTH, kv.BAD_LENGTH]


def test_random_rounds_conserve_pages():
    rng = np.random.default_rng(0)
    nb, B, mb = 200, 12, 40
    tables, stack, F = _fresh(nb, B, mb)
    ctx = [0] * B
    for _ in range(30):
        draft = rng.integers(0, 9, size=B).tolist()
        F, codes = kv.reserve_append(tables, stack, F, ctx, draft, nb)
        acc = [int(rng.integers(0, d + 1)) if codes[r] == 0 else 0 for r, d in enumerate(draft)]
        served = [codes[r] == 0 for r in range(B)]
        F, _ = kv.commit(tables, stack, F, ctx, [d if s else -1 for d, s in zip(draft, served)], acc)
        used = [p for row in tables for p in row if p >= 0]
        assert sorted(used + stack[:F]) == list(range(nb))
        for r in range(B):   # a request holds exactly the pages of its committed prefix
            assert sum(p >= 0 for p in tables[r]) == (ctx[r] + 15) // 16
