"""GPU parity: the copy-on-write page pool through the C ABI vs the oracle.

The same operations run on the GPU pool and on the oracle's sequential
PagePool.  Which page ids the GPU hands out depends on scheduling, so what is
compared is what the definition fixes: the bytes every table addresses, the
number of free pages, holder counts equal to the number of table slots
holding each page (counted here from the GPU's own tables), the free stack
equal to the pages held by nobody, and -- for KV sessions forked by sharing
pages -- whole PCS1 records equal to the oracle's, with the parent's record
unchanged by the child's writes (I3).
"""
from collections import Counter

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs

pytestmark = pytest.mark.gpu


def _gather(pages, table):
    ids = table.reshape(-1)
    ids = ids[ids >= 0].long()
    return pages[ids].reshape(-1).cpu().numpy()


def _check_state(pool, tables):
    free, counts, free_ids = pool.query()
    held = Counter(p for t in tables for p in t.reshape(-1).cpu().tolist() if p >= 0)
    want = np.zeros(pool.n_pages, dtype=np.uint32)
    for p, c in held.items():
        want[p] = c
    assert np.array_equal(counts, want)
    assert sorted(free_ids.tolist()) == [p for p in range(pool.n_pages) if want[p] == 0]
    return free


def _write(dev_pages, o_pool, gt, ot, entries, rnd):
    """The same new bytes into the pages at `entries` of both tables."""
    for e in entries:
        data = rnd.integers(0, 256, o_pool.data.shape[1], dtype=np.uint8)
        o_pool.data[ot.reshape(-1)[e]] = data
        dev_pages[int(gt.reshape(-1)[e])] = torch.from_numpy(data).to(dev_pages.device)


@pytest.mark.parametrize("seed", range(6))
def test_pool_random_sequences_match_oracle(ctx, dev, seed):
    rnd = np.random.default_rng(seed)
    n_pages, page_bytes = 3000, 272
    pages = torch.zeros(n_pages, page_bytes, dtype=torch.uint8, device=dev)
    pool = pcs.Pool(ctx, pages)
    op = oracle.PagePool(n_pages, page_bytes)
    gts, ots = [], []
    for _ in range(3):
        k = int(rnd.integers(1, 40))
        gt, ot = pool.alloc(k), op.alloc(k)
        _write(pages, op, gt, ot, range(k), rnd)
        gts.append(gt)
        ots.append(ot)
    for step in range(40):
        kind = int(rnd.integers(0, 4))
        if kind == 0:                                  # fork
            i = int(rnd.integers(0, len(gts)))
            gts.append(pool.share(gts[i]))
            ots.append(op.share(ots[i]))
        elif kind == 1:                                # copy leg + write
            i = int(rnd.integers(0, len(gts)))
            ent = rnd.choice(gts[i].numel(), size=int(rnd.integers(1, gts[i].numel() + 1)),
                             replace=False).astype(np.int32)
            pool.prepare_write(gts[i], torch.from_numpy(ent).to(dev))
            op.prepare_write(ots[i], ent)
            torch.cuda.synchronize()
            _write(pages, op, gts[i], ots[i], ent.tolist(), rnd)
        elif kind == 2 and len(gts) > 1:               # drop a table
            i = int(rnd.integers(0, len(gts)))
            pool.release(gts.pop(i))
            op.release(ots.pop(i))
        elif kind == 3 and len(op.free) > 50:          # a new table
            k = int(rnd.integers(1, 30))
            gt, ot = pool.alloc(k), op.alloc(k)
            _write(pages, op, gt, ot, range(k), rnd)
            gts.append(gt)
            ots.append(ot)
        ctx.sync()
        assert _check_state(pool, gts) == len(op.free), step
        for gt, ot in zip(gts, ots):
            assert np.array_equal(_gather(pages, gt), op.gather(ot)), step
    for gt in gts:
        pool.release(gt)
    ctx.sync()
    assert _check_state(pool, []) == n_pages
    pool.destroy()


@pytest.mark.parametrize("holders,writers", [(2, 2), (4, 2), (4, 4), (8, 8)])
def test_pool_many_holders_in_one_call(ctx, dev, holders, writers):
    # One table tensor holding several forks of the same pages: all but one
    # holder of each page copy, whichever the GPU lets keep it.
    pages = torch.zeros(512, 64, dtype=torch.uint8, device=dev)
    pool = pcs.Pool(ctx, pages)
    op = oracle.PagePool(512, 64)
    rnd = np.random.default_rng(holders * 10 + writers)
    g0, o0 = pool.alloc(33), op.alloc(33)
    _write(pages, op, g0, o0, range(33), rnd)
    gs = [g0] + [pool.share(g0) for _ in range(holders - 1)]
    os_ = [o0] + [op.share(o0) for _ in range(holders - 1)]
    big = torch.stack(gs[:writers]).contiguous()
    obig = np.stack(os_[:writers])
    pool.prepare_write(big)
    op.prepare_write(obig)
    ctx.sync()
    gs = [big[i] for i in range(writers)] + gs[writers:]
    assert _check_state(pool, gs) == len(op.free)
    copies = (writers if writers < holders else writers - 1) * 33
    assert op.copies == copies and len(op.free) == 512 - 33 - copies
    for g in gs:
        assert np.array_equal(_gather(pages, g), op.gather(o0))
    # After the copy leg every written slot's page is its own.
    _, counts, _ = pool.query()
    assert (counts[big.reshape(-1).long().cpu().numpy()] == 1).all()
    pool.destroy()


def test_kv_fork_by_sharing_pages(ctx, dev):
    # KV sessions whose K and V pages live in one pool: fork every session by
    # sharing its page tables, append a token to each child (copy leg on the
    # ring page it writes), and compare whole records with the oracle.
    S, layers, pr, heads, hd, window = 3, 2, 16, 4, 16, 64
    per = window // pr
    n_pages = 2 * S * layers * per * 2 + 8
    rb = heads * hd * 2
    rnd = np.random.default_rng(5)
    pages = torch.zeros(n_pages, pr, heads, hd, dtype=torch.bfloat16, device=dev)
    pool = pcs.Pool(ctx, pages)
    op = oracle.PagePool(n_pages, pr * rb)
    pages_u8 = pages.view(torch.uint8).view(n_pages, pr * rb)
    ring = [int(x) for x in rnd.integers(0, window, S)]
    meta = [rnd.integers(0, 2**40, 4).astype(np.int64) for _ in range(S)]
    par_g, par_o = [], []
    for s in range(S):
        kt, ko = pool.alloc(layers * per), op.alloc(layers * per)
        vt, vo = pool.alloc(layers * per), op.alloc(layers * per)
        _write(pages_u8, op, kt, ko, range(layers * per), rnd)
        _write(pages_u8, op, vt, vo, range(layers * per), rnd)
        par_g.append((kt.view(layers, per), vt.view(layers, per)))
        par_o.append((ko.reshape(layers, per), vo.reshape(layers, per)))

    def g_sess(s, tabs, sid):
        return pcs.kv_session(sid, torch.from_numpy(meta[s]).to(dev), pages, pages, tabs[0],
                              ring[s], window, v_page_table=tabs[1])

    def o_rec(s, tabs, sid):
        return oracle.pack(oracle.kv_session(sid, meta[s], op.data, op.data, tabs[0], ring[s],
                                             window, pr, rb, v_page_table=tabs[1]))

    snaps0 = ctx.checkpoint([g_sess(s, par_g[s], s) for s in range(S)])
    before = [ctx.record(x).numpy() for x in snaps0]
    for x in snaps0:
        ctx.delete(x)
    for s in range(S):
        assert np.array_equal(before[s], o_rec(s, par_o[s], s))
    ch_g = [(pool.share(k), pool.share(v)) for k, v in par_g]
    ch_o = [(op.share(k), op.share(v)) for k, v in par_o]
    ctx.sync()
    free_after_fork = pool.query()[0]
    assert free_after_fork == len(op.free) == n_pages - 2 * S * layers * per
    # Each child appends one token at its ring slot `ring` (oldest row).
    for s in range(S):
        page_idx = ring[s] // pr
        ent = np.array([l * per + page_idx for l in range(layers)], dtype=np.int32)
        for t in (0, 1):
            pool.prepare_write(ch_g[s][t], torch.from_numpy(ent).to(dev))
            op.prepare_write(ch_o[s][t], ent)
        torch.cuda.synchronize()
        row = ring[s] % pr
        for t in (0, 1):
            for e in ent.tolist():
                new = rnd.integers(0, 256, rb, dtype=np.uint8)
                q_o = int(ch_o[s][t].reshape(-1)[e])
                op.data[q_o, row * rb:(row + 1) * rb] = new
                q_g = int(ch_g[s][t].reshape(-1)[e])
                pages_u8[q_g, row * rb:(row + 1) * rb] = torch.from_numpy(new).to(dev)
    ctx.sync()
    assert pool.query()[0] == len(op.free) == free_after_fork - S * layers * 2
    snaps = ctx.checkpoint([g_sess(s, par_g[s], s) for s in range(S)] +
                           [g_sess(s, ch_g[s], 10 + s) for s in range(S)])
    for s in range(S):
        assert np.array_equal(ctx.record(snaps[s]).numpy(), before[s])      # I3
        assert np.array_equal(ctx.record(snaps[S + s]).numpy(), o_rec(s, ch_o[s], 10 + s))
        assert not np.array_equal(ctx.record(snaps[S + s]).numpy()[256:], before[s][256:])
    for x in snaps:
        ctx.delete(x)
    pool.destroy()


def test_pool_errors_are_reported_and_state_stays_consistent(ctx, dev):
    pages = torch.zeros(10, 32, dtype=torch.uint8, device=dev)
    pool = pcs.Pool(ctx, pages)
    a = pool.alloc(6)
    b = pool.share(a)
    ctx.sync()
    # The copy leg needs 6 pages and 4 are free: 4 slots copy, 2 keep sharing.
    pool.prepare_write(b)
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    assert e.value.status == pcs.PCS_E_NOMEM
    assert _check_state(pool, [a, b]) == 0
    assert int((a != b).sum()) == 4
    # Alloc from an empty pool: -1 ids and an error.
    c = pool.alloc(2)
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    assert e.value.status == pcs.PCS_E_NOMEM and c.cpu().tolist() == [-1, -1]
    # Ids outside the pool are skipped and reported.
    bad = torch.tensor([3, 10, -1, 99], dtype=torch.int32, device=dev)
    pool.share(bad)
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    assert e.value.status == pcs.PCS_E_RANGE
    pool.release(bad[:1])  # undo the one valid share
    # Releasing more often than held is refused per page.
    pool.release(a)
    pool.release(b)
    ctx.sync()
    assert _check_state(pool, []) == 10
    pool.release(a[:1])
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    assert e.value.status == pcs.PCS_E_INVAL
    assert _check_state(pool, []) == 10
    # Empty slots are skipped everywhere.
    t = torch.tensor([-1, -1], dtype=torch.int32, device=dev)
    pool.share(t)
    pool.prepare_write(t)
    pool.release(t)
    ctx.sync()
    pool.destroy()
    with pytest.raises(pcs.PcsError) as e:
        pool.alloc(1)
    assert e.value.status == pcs.PCS_E_HANDLE
