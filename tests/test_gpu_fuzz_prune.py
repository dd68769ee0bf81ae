"""GPU: seeded random relevance-pruning calls against the oracle.

Each trial draws a call of 1 to 40 banks: key widths from 8 to 1,536 (every
score kernel: one, two and four 16-byte segments per lane and the generic
loop), fp16, bf16 or both in one call, bank sizes from 0 up to 600 or up to
5,000 entries (both top-k paths: keys held in registers up to 4,096 entries,
re-read above), some banks drawn from a handful of distinct keys (runs of
exact ties at the threshold), the fixed, fraction and budget k-rules, and
packed or 16-byte aligned kept lists.  The counts, the offsets, every score
(bit for bit) and every kept list must equal the oracle's."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs
from helpers import np_view

pytestmark = pytest.mark.gpu

DIMS = [8, 16, 64, 128, 256, 264, 512, 520, 1024, 1032, 1536]


@pytest.mark.parametrize("trial", range(16))
def test_random_prune_calls(ctx, dev, trial):
    rnd = np.random.default_rng(4000 + trial)
    g = torch.Generator().manual_seed(4000 + trial)
    nb = int(rnd.integers(1, 41))
    D = int(DIMS[trial % len(DIMS)] if trial < len(DIMS) else rnd.choice(DIMS))
    mixed = trial % 5 == 4
    big = trial % 4 == 3
    n = [int(x) for x in rnd.integers(0, 5000 if big else 600, nb)]
    one_dt = torch.float16 if trial % 2 == 0 else torch.bfloat16
    keys, qs = [], []
    for i in range(nb):
        dt = (torch.float16 if rnd.random() < 0.5 else torch.bfloat16) if mixed else one_dt
        qs.append(torch.randn(D, generator=g).to(dt))
        if n[i] > 0 and rnd.random() < 0.3:
            pool = torch.randn(int(rnd.integers(1, 6)), D, generator=g).to(dt)
            keys.append(pool[torch.randint(0, pool.shape[0], (n[i],), generator=g)].contiguous())
        else:
            keys.append(torch.randn(n[i], D, generator=g).to(dt))
    entry = 2 * D + int(rnd.choice([0, 16, 2048]))
    align = int(rnd.choice([0, 1, 4]))
    rule = ["fixed", "fraction", "budget"][trial % 3]
    if rule == "fixed":
        k_max = int(rnd.integers(0, 700))
        params = ctx.params(pcs.PCS_K_FIXED, k_max=k_max, kept_align=align)
        want_k = oracle.k_fixed(n, k_max)
    elif rule == "fraction":
        frac = float(rnd.random())
        params = ctx.params(pcs.PCS_K_FRACTION, fraction=frac, kept_align=align)
        want_k = oracle.k_fraction(n, frac)
    else:
        budget = int(sum(n) * entry * rnd.random())
        params = ctx.params(pcs.PCS_K_BUDGET, budget=budget, kept_align=align)
        want_k = oracle.k_budget(n, entry, budget)
    kd = [k.to(dev) for k in keys]
    qd = [q.to(dev) for q in qs]
    banks = ctx.banks_array(kd, qd, entry)
    ks = ctx.prune_counts(banks, nb, params)
    assert ks == want_k.tolist()
    a = 4 if align == 4 else 1
    off = np.concatenate([[0], np.cumsum([(k + a - 1) // a * a for k in ks])]).astype(np.int64)
    kept = torch.full((max(int(off[-1]), 1),), -7, dtype=torch.int32, device=dev)
    koff = torch.empty(nb + 1, dtype=torch.int32, device=dev)
    scores = torch.empty(max(sum(n), 1), dtype=torch.float32, device=dev)
    ctx.prune(banks, nb, params, kept, koff, scores)
    ctx.sync()
    assert koff.cpu().numpy().tolist() == off.tolist()
    sc_h, kept_h = scores.cpu().numpy(), kept.cpu().numpy()
    eo = 0
    for i in range(nb):
        s32 = oracle.scores(np_view(qs[i]), np_view(keys[i]))
        got = sc_h[eo:eo + n[i]]
        assert np.array_equal(got.view(np.uint32), s32.view(np.uint32)), (trial, i)
        assert kept_h[off[i]:off[i] + ks[i]].tolist() == oracle.topk(s32, ks[i]).tolist(), (trial, i)
        eo += n[i]
