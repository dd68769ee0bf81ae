"""Pins of the oracle's copy-on-write page pool (CPU only).

Sec. 3 (I3): a child's continuation is independent of its parent's, and the
mechanism realises this by copy-on-write; Sec. 7.3: blocks carry reference
counts and their copy leg fires on the first write.  The pins: reference
counts always equal the number of table slots that hold a page (counted here
by brute force), the free pages are exactly those held by nobody, sharing and
the copy leg never change what any table addresses, a write after the copy
leg is invisible to every other table (I3 both ways), and the number of
copies is the one the definition fixes.
"""
from collections import Counter

import numpy as np
import pytest

import oracle


def _check_invariants(pool, tables):
    held = Counter(p for t in tables for p in t.reshape(-1).tolist() if p >= 0)
    for p in range(pool.rc.size):
        assert pool.rc[p] == held.get(p, 0), p
    assert len(set(pool.free)) == len(pool.free)
    assert set(pool.free) == {p for p in range(pool.rc.size) if held.get(p, 0) == 0}


def _fill(pool, table, rnd):
    for p in table.reshape(-1).tolist():
        if p >= 0:
            pool.data[p] = rnd.integers(0, 256, pool.data.shape[1], dtype=np.uint8)


@pytest.mark.parametrize("seed", range(25))
def test_random_sequences_keep_counts_and_contents(seed):
    rnd = np.random.default_rng(seed)
    pool = oracle.PagePool(400, 32)
    tables = []
    for _ in range(3):
        t = pool.alloc(int(rnd.integers(1, 20))).reshape(1, -1)
        _fill(pool, t, rnd)
        tables.append(t)
    for step in range(60):
        op = rnd.integers(0, 4)
        if op == 0 and tables:            # fork a table
            src = tables[int(rnd.integers(0, len(tables)))]
            before = pool.gather(src)
            tables.append(pool.share(src))
            assert np.array_equal(pool.gather(tables[-1]), before)
        elif op == 1 and tables:          # copy leg on some entries, then write them
            t = tables[int(rnd.integers(0, len(tables)))]
            ent = rnd.choice(t.size, size=int(rnd.integers(1, t.size + 1)), replace=False)
            others = [(o, pool.gather(o)) for o in tables if o is not t]
            before = pool.gather(t)
            pool.prepare_write(t, ent)
            assert np.array_equal(pool.gather(t), before)
            for e in ent.tolist():
                p = int(t.reshape(-1)[e])
                assert pool.rc[p] == 1  # written pages are held by this entry alone
                pool.data[p] = rnd.integers(0, 256, pool.data.shape[1], dtype=np.uint8)
            for o, g in others:           # I3: nobody else sees the writes
                assert np.array_equal(pool.gather(o), g)
        elif op == 2 and len(tables) > 1:  # drop a table
            t = tables.pop(int(rnd.integers(0, len(tables))))
            pool.release(t)
        elif op == 3 and len(pool.free) > 5:
            t = pool.alloc(int(rnd.integers(1, 5))).reshape(1, -1)
            _fill(pool, t, rnd)
            tables.append(t)
        _check_invariants(pool, tables)
    for t in tables:
        pool.release(t)
    assert len(pool.free) == 400 and not pool.rc.any()


def test_fork_independence_both_ways():
    rnd = np.random.default_rng(1)
    pool = oracle.PagePool(64, 16)
    parent = pool.alloc(8)
    _fill(pool, parent, rnd)
    g_parent = pool.gather(parent)
    child = pool.share(parent)
    assert len(pool.free) == 56  # a fork moves no bytes and takes no page
    pool.prepare_write(child, [2, 5])
    for e in (2, 5):
        pool.data[child[e]] ^= 0xFF
    assert np.array_equal(pool.gather(parent), g_parent)
    g_child = pool.gather(child)
    pool.prepare_write(parent, None)
    pool.data[parent[5]] = 7
    assert np.array_equal(pool.gather(child), g_child)
    # Entry 5 was copied by the child, so the parent's page 5 was already its
    # own: its second copy leg took pages only for the 6 entries still shared.
    assert pool.copies == 2 + 6


@pytest.mark.parametrize("holders,writers", [(2, 1), (2, 2), (5, 3), (5, 5), (1, 1)])
def test_copy_count(holders, writers):
    pool = oracle.PagePool(16, 8)
    t0 = pool.alloc(1)
    ts = [t0] + [pool.share(t0) for _ in range(holders - 1)]
    for t in ts[:writers]:
        pool.prepare_write(t)
    # Each writer copies while others still hold the page; the last holder keeps it.
    assert pool.copies == (writers if writers < holders else writers - 1)
    _check_invariants(pool, ts)


def test_empty_slots_and_errors():
    pool = oracle.PagePool(4, 8)
    t = np.array([-1, 0, -1], dtype=np.int32)
    with pytest.raises(oracle.PoolError):
        pool.release([0])
    a = pool.alloc(4)
    assert a.tolist() == [0, 1, 2, 3]
    with pytest.raises(oracle.PoolError):
        pool.alloc(1)
    s = pool.share(t)
    assert pool.rc.tolist() == [2, 1, 1, 1]
    with pytest.raises(oracle.PoolError):
        pool.prepare_write(s)  # page 0 is shared and the pool is full
