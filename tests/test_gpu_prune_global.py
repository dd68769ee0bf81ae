"""GPU parity: one relevance threshold across all banks under a byte budget.

pcs_prune_global through the C ABI against the oracle on the same seeded
banks: scores bit-equal to the oracle's fixed-order fp32 score, kept sets and
bank offsets identical, across several 4096-entry tiles with a ragged tail,
with uniform and mixed entry sizes (the two select paths), empty banks at
either end and in the middle, exact ties across banks, mixed key types and
keys wider than 1024 (the first digit binned after the score kernel), and
budgets that keep nothing, one entry, a fraction, all but one, and all.  The same population
split into two parts (two threads, two contexts, the histograms summed on the
host each pass, as ranks would all-reduce them) gives each part its share of
the one-population answer.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_view

pytestmark = pytest.mark.gpu


def _oracle_scores(keys, qs):
    return np.concatenate([oracle.scores(np_view(q), np_view(k)) if k.shape[0] else
                           np.zeros(0, np.float32) for k, q in zip(keys, qs)])


def _run(ctx, dev, keys, qs, E, budget, want_scores=True):
    n = len(keys)
    banks = ctx.banks_array(keys, qs, E)
    total = sum(k.shape[0] for k in keys)
    kept = torch.full((max(total, 1),), -7, dtype=torch.int32, device=dev)
    koff = torch.full((n + 1,), -7, dtype=torch.int32, device=dev)
    scores = torch.empty(max(total, 1), dtype=torch.float32, device=dev) if want_scores else None
    ctx.prune_global(banks, n, budget, kept, koff, scores)
    ctx.sync()
    koff_h = koff.cpu().numpy()
    kept_h = kept.cpu().numpy()[:koff_h[-1]]
    return kept_h, koff_h, (scores.cpu().numpy()[:total] if want_scores else None)


def _check(ctx, dev, keys, qs, E, budgets):
    s32 = _oracle_scores(keys, qs)
    n = [k.shape[0] for k in keys]
    Eb = [E] * len(n) if isinstance(E, int) else E
    for B in budgets:
        kept, koff, sc = _run(ctx, dev, keys, qs, E, B)
        assert np.array_equal(sc.view(np.uint32), s32.view(np.uint32))
        want, woff = oracle.prune_global(s32, n, Eb, B)
        assert koff.tolist() == woff.tolist(), B
        assert kept.tolist() == want.tolist(), B


def _views(b, dev):
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]].to(dev) for s in range(b.sessions)]
    qs = [b.queries[s].to(dev) for s in range(b.sessions)]
    return keys, qs


def test_global_threshold_uniform_bytes(ctx, dev):
    # ~6,000 entries: two 4096-entry tiles, the second ragged.
    b = synth.banks(301, 40, 1, 300, 256, torch.float16, (8,), torch.uint8)
    keys, qs = _views(b, dev)
    E = 512 + 8
    T = sum(b.n) * E
    _check(ctx, dev, keys, qs, E, [0, E - 1, E, 7 * E + 3, T // 10, T // 2, T - E, T - 1, T,
                                   T + 1, 2 * T])


def test_global_threshold_mixed_bytes_and_empty_banks(ctx, dev):
    b = synth.banks(302, 30, 0, 700, 128, torch.bfloat16, (8,), torch.uint8)
    keys, qs = _views(b, dev)
    # Empty banks first, in the middle and last.
    D = keys[0].shape[1]
    empty = torch.empty(0, D, dtype=keys[0].dtype, device=dev)
    keys = [empty, empty] + keys[:10] + [empty] + keys[10:] + [empty, empty]
    qs = [qs[0], qs[1]] + qs[:10] + [qs[2]] + qs[10:] + [qs[3], qs[4]]
    rnd = np.random.default_rng(3)
    E = [int(x) for x in rnd.integers(0, 5000, len(keys))]
    E[5] = 0  # free entries still take their place in the order
    T = sum(k.shape[0] * e for k, e in zip(keys, E))
    _check(ctx, dev, keys, qs, E, [0, 1, T // 7, T // 3, T // 2, T - 1, T])


def test_global_threshold_ties_across_banks(ctx, dev):
    # Zero keys score 0 everywhere and duplicated keys tie exactly: the order
    # falls through to bank, then index -- the low digit passes decide.
    D = 64
    g = torch.Generator().manual_seed(8)
    q = torch.randn(D, generator=g).half()
    base = torch.randn(3, D, generator=g).half()
    banks_k = []
    for s in range(9):
        parts = [torch.zeros(500 + 37 * s, D).half(), base, base[:1].repeat(4, 1)]
        banks_k.append(torch.cat(parts).to(dev))
    qs = [q.to(dev)] * 9
    E = 96
    T = sum(k.shape[0] for k in banks_k) * E
    _check(ctx, dev, banks_k, qs, E, [0, E, 5 * E, 30 * E + 5, T // 2 + 17 * E, T - E, T])
    _check(ctx, dev, banks_k, qs, [96, 1, 300, 96, 7, 96, 1000, 2, 96],
           [0, 1000, 12345, 200000, 10**9])


def test_global_threshold_scores_optional_and_no_entries(ctx, dev):
    b = synth.banks(303, 7, 1, 50, 64, torch.float16, (8,), torch.uint8)
    keys, qs = _views(b, dev)
    s32 = _oracle_scores(keys, qs)
    kept, koff, _ = _run(ctx, dev, keys, qs, 100, sum(b.n) * 40, want_scores=False)
    want, woff = oracle.prune_global(s32, b.n, 100, sum(b.n) * 40)
    assert koff.tolist() == woff.tolist() and kept.tolist() == want.tolist()
    empty = torch.empty(0, 64, dtype=torch.float16, device=dev)
    kept, koff, _ = _run(ctx, dev, [empty] * 3, qs[:3], 100, 10, want_scores=False)
    assert koff.tolist() == [0, 0, 0, 0]


def test_global_threshold_unaligned_scores(ctx, dev):
    # A scores buffer that starts 4 bytes past a 16-byte boundary: the scans
    # read it one float at a time.
    b = synth.banks(304, 9, 100, 900, 64, torch.float16, (8,), torch.uint8)
    keys, qs = _views(b, dev)
    total = sum(b.n)
    banks = ctx.banks_array(keys, qs, 200)
    buf = torch.zeros(total + 4, dtype=torch.float32, device=dev)
    scores = buf[1:1 + total]
    kept = torch.empty(total, dtype=torch.int32, device=dev)
    koff = torch.empty(len(keys) + 1, dtype=torch.int32, device=dev)
    B = total * 200 * 2 // 5
    ctx.prune_global(banks, len(keys), B, kept, koff, scores)
    ctx.sync()
    s32 = _oracle_scores(keys, qs)
    assert np.array_equal(scores.cpu().numpy().view(np.uint32), s32.view(np.uint32))
    want, woff = oracle.prune_global(s32, b.n, 200, B)
    assert koff.cpu().tolist() == woff.tolist()
    assert kept.cpu().tolist()[:woff[-1]] == want.tolist()


def test_global_threshold_keeps_relevant_sessions(ctx, dev):
    # Against the same-fraction rule: a bank aligned with its query keeps
    # more under the global threshold.
    D = 128
    g = torch.Generator().manual_seed(12)
    q = torch.randn(D, generator=g)
    near = (q[None] + 0.3 * torch.randn(200, D, generator=g)).half()
    far = torch.randn(200, D, generator=g).half()
    keys = [near.to(dev), far.to(dev)]
    qs = [q.half().to(dev)] * 2
    kept, koff, _ = _run(ctx, dev, keys, qs, 10, 2000)
    assert koff.tolist() == [0, 200, 200]


@pytest.mark.parametrize("mixed_bytes", [False, True])
def test_global_threshold_mixed_key_types(ctx, dev, mixed_bytes):
    # fp16 and bf16 banks together (and, below, keys wider than 1024): the
    # score kernel takes no digit pass, so the first is binned after it.
    g = torch.Generator().manual_seed(21)
    D = 96
    keys, qs = [], []
    for s in range(14):
        dt = torch.float16 if s % 2 else torch.bfloat16
        n = int(torch.randint(0, 900, (1,), generator=g))
        keys.append(torch.randn(n, D, generator=g).to(dt).to(dev))
        qs.append(torch.randn(D, generator=g).to(dt).to(dev))
    E = [int(x) for x in np.random.default_rng(4).integers(1, 3000, 14)] if mixed_bytes else 700
    Eb = E if mixed_bytes else [E] * 14
    T = sum(k.shape[0] * e for k, e in zip(keys, Eb))
    _check(ctx, dev, keys, qs, E, [0, 1, T // 9, T // 2, T - 1, T])


def test_global_threshold_wide_keys(ctx, dev):
    g = torch.Generator().manual_seed(22)
    D = 1536
    keys = [torch.randn(int(n), D, generator=g).half().to(dev) for n in (300, 0, 1200, 77)]
    qs = [torch.randn(D, generator=g).half().to(dev) for _ in range(4)]
    T = sum(k.shape[0] for k in keys) * 50
    _check(ctx, dev, keys, qs, 50, [0, 50, T // 3, T - 50, T])


def _split_run(dev, keys, qs, E, budget, cut):
    """Two parts (banks [:cut] and [cut:]) run as two threads with their own
    contexts and streams; the exchange sums the histograms through a barrier."""
    import threading
    parts = [(keys[:cut], qs[:cut], E[:cut]), (keys[cut:], qs[cut:], E[cut:])]
    base = [0, sum(k.shape[0] for k in keys[:cut])]
    barrier = threading.Barrier(2)
    slot_c, slot_b, out, errs = [None, None], [None, None], [None, None], []

    def worker(r):
        try:
            pk, pq, pe = parts[r]
            with pcs.Context(0) as c:
                s = torch.cuda.Stream(device=dev)
                banks = c.banks_array(pk, pq, pe) if pk else (pcs.pcs_bank * 1)()
                total = sum(k.shape[0] for k in pk)
                kept = torch.full((max(total, 1),), -7, dtype=torch.int32, device=dev)
                koff = torch.full((len(pk) + 1,), -7, dtype=torch.int32, device=dev)

                def ex(cnt, byt):
                    slot_c[r], slot_b[r] = cnt.copy(), byt.copy()
                    barrier.wait(60)
                    tc, tb = slot_c[0] + slot_c[1], slot_b[0] + slot_b[1]
                    barrier.wait(60)
                    cnt[:] = tc
                    byt[:] = tb
                c.prune_global_part(banks, len(pk), budget, base[r], ex, kept, koff, stream=s)
                s.synchronize()
                ko = koff.cpu().numpy()
                out[r] = (kept.cpu().numpy()[:ko[-1]], ko)
        except BaseException as e:  # surfaced below
            errs.append(e)
            barrier.abort()

    ts = [threading.Thread(target=worker, args=(r,)) for r in range(2)]
    for t in ts:
        t.start()
    for t in ts:
        t.join(300)
    assert not errs, errs
    return out


@pytest.mark.parametrize("budget_frac", [0.0, 0.3, 0.62, 1.0])
def test_global_threshold_split_across_parts(dev, budget_frac):
    b = synth.banks(310, 30, 0, 600, 128, torch.bfloat16, (8,), torch.uint8)
    keys, qs = _views(b, dev)
    rnd = np.random.default_rng(11)
    E = [int(x) for x in rnd.integers(1, 4000, len(keys))]
    T = sum(k.shape[0] * e for k, e in zip(keys, E))
    B = int(T * budget_frac)
    s32 = _oracle_scores(keys, qs)
    want, woff = oracle.prune_global(s32, [k.shape[0] for k in keys], E, B)
    for cut in (12, 0):  # the second split gives part 0 no banks at all
        got = _split_run(dev, keys, qs, E, B, cut)
        for r, (lo, hi) in enumerate(((0, cut), (cut, len(keys)))):
            kept, ko = got[r]
            assert ko.tolist() == (woff[lo:hi + 1] - woff[lo]).tolist(), (cut, r)
            assert kept.tolist() == want[woff[lo]:woff[hi]].tolist(), (cut, r)


def test_global_threshold_one_part_equals_whole(ctx, dev):
    b = synth.banks(311, 25, 1, 400, 64, torch.float16, (8,), torch.uint8)
    keys, qs = _views(b, dev)
    banks = ctx.banks_array(keys, qs, 300)
    total = sum(b.n)
    B = total * 300 // 3
    kept = torch.empty(total, dtype=torch.int32, device=dev)
    koff = torch.empty(len(keys) + 1, dtype=torch.int32, device=dev)
    ctx.prune_global_part(banks, len(keys), B, 0, lambda c, x: None, kept, koff)
    ctx.sync()
    want, woff = oracle.prune_global(_oracle_scores(keys, qs), b.n, 300, B)
    assert koff.cpu().tolist() == woff.tolist()
    assert kept.cpu().tolist()[:woff[-1]] == want.tolist()
