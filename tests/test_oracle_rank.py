"""Pins of the oracle's relevance score, ranking and k-rules (CPU only).

The paper ranks bank frames by relevance to the return viewpoint and prunes
every bank to the same fraction when the host budget binds (Sec. 5, Sec. 7.5,
Table tab:keepfrac); it gives no formula.  The reading is a cosine score
(fp32, fixed order -- the precision that decides the kept set), ranking by
(score desc, entry index asc), selection rather than merging (Sec. 9).
"""
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf16_bits(x):
    return torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).view(torch.int16).numpy().view(
        np.uint16)


def _rand_keys(seed, n, D, dtype):
    rnd = np.random.default_rng(seed)
    if dtype == "f16":
        return (rnd.standard_normal(D).astype(np.float16),
                rnd.standard_normal((n, D)).astype(np.float16))
    return _bf16_bits(rnd.standard_normal(D)), _bf16_bits(rnd.standard_normal((n, D)))


def _as_f64(a):
    if a.dtype == np.float16:
        return a.astype(np.float64)
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("dtype,D", [("f16", 256), ("bf16", 512), ("f16", 8), ("bf16", 40)])
def test_score_matches_numpy_cosine(dtype, D):
    q, k = _rand_keys(D, 300, D, dtype)
    s32, s64 = oracle.scores(q, k, want64=True)
    qd, kd = _as_f64(q), _as_f64(k)
    ref = kd @ qd / (np.linalg.norm(kd, axis=1) * np.linalg.norm(qd))
    np.testing.assert_allclose(s64, ref, rtol=1e-12, atol=1e-15)
    # The fp32 fixed-order score is within the 1e-3 relative tolerance.
    np.testing.assert_allclose(s32, ref, rtol=1e-3, atol=1e-6)


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_score_closed_forms(dtype):
    q, k = _rand_keys(7, 4, 256, dtype)
    qrow = q[None, :]
    s = oracle.scores(q, qrow)
    assert abs(s[0] - 1.0) <= 2 ** -22
    neg = (-_as_f64(q)).astype(np.float16) if dtype == "f16" else (q ^ np.uint16(0x8000))
    assert abs(oracle.scores(q, neg[None, :])[0] + 1.0) <= 2 ** -22
    # Scaling a key by 2 is exact at every step, so the fp32 score is identical.
    if dtype == "f16":
        k2 = (k.astype(np.float32) * 2).astype(np.float16)
    else:
        k2 = _bf16_bits((_as_f64(k) * 2))
    assert np.array_equal(oracle.scores(q, k), oracle.scores(q, k2))
    # Orthogonal unit vectors and a zero key.
    e0 = np.zeros(256, np.float16); e0[0] = 1
    e1 = np.zeros(256, np.float16); e1[200] = 1
    assert oracle.scores(e0, e1[None, :])[0] == 0.0
    assert oracle.scores(e0, np.zeros((1, 256), np.float16))[0] == 0.0


def _brute_topk(scores, k):
    # Independent: Python's sort on (-score, index), NaN last, -0 == +0.
    def rank_key(i):
        s = float(scores[i])
        return (1, 0.0, i) if np.isnan(s) else (0, -s, i)
    order = sorted(range(len(scores)), key=rank_key)
    return sorted(order[:min(k, len(scores))])


@pytest.mark.parametrize("seed", range(30))
def test_topk_matches_brute_force(seed):
    rnd = np.random.default_rng(seed)
    n = int(rnd.integers(1, 12))
    # Few distinct values so that ties are common, plus signed zeros and NaN.
    pool = np.array([0.5, -0.25, 0.0, -0.0, 1.0, np.nan, 0.5], dtype=np.float32)
    s = pool[rnd.integers(0, pool.size, n)]
    for k in range(0, n + 2):
        assert oracle.topk(s, k).tolist() == _brute_topk(s, k), (s, k)


def test_topk_ties_go_to_lower_index():
    s = np.full(10, 0.3, dtype=np.float32)
    assert oracle.topk(s, 4).tolist() == [0, 1, 2, 3]


def test_key64_order():
    vals = [-np.inf, -1.0, -1e-30, 0.0, 1e-30, 1.0, np.inf]
    keys = [oracle.ord32(v) for v in vals]
    assert keys == sorted(keys) and len(set(keys)) == len(keys)
    assert oracle.ord32(-0.0) == oracle.ord32(0.0)
    assert oracle.ord32(float("nan")) == 0 < oracle.ord32(-np.inf)
    assert oracle.key64(0.5, 3) > oracle.key64(0.5, 4) > oracle.key64(0.25, 0)


def test_fraction_rule_reproduces_keepfrac_table():
    # Table tab:keepfrac: frames kept of ~21 at each keep fraction.
    rows = []
    with open(os.path.join(GOLDEN, "keepfrac_table.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                frac, kept = line.split()
                rows.append((float(frac), int(kept)))
    assert len(rows) == 5
    for frac, kept in rows:
        assert oracle.k_fraction([21], frac).tolist() == [kept], frac


def test_fixed_rule():
    assert oracle.k_fixed([1, 127, 128, 129, 512], 128).tolist() == [1, 127, 128, 128, 128]


def test_budget_rule_keeps_all_when_budget_does_not_bind():
    n = [10, 20, 30]
    assert oracle.k_budget(n, 3072, 60 * 3072).tolist() == n
    assert oracle.k_budget(n, 3072, 10**12).tolist() == n


def test_budget_rule_closed_form_and_inequality():
    rnd = np.random.default_rng(1)
    n = rnd.integers(256, 4097, 2048).astype(np.int32)
    E = 1024 + 2048
    B = 8 << 30
    k = oracle.k_budget(n, E, B)
    T = int(n.astype(np.int64).sum()) * E
    assert T > B
    # Same fraction B/T for every bank, rounded down; total within budget.
    for ni, ki in zip(n.tolist(), k.tolist()):
        assert ki == (ni * B) // T
    assert int(k.astype(np.int64).sum()) * E <= B
    assert int(k.astype(np.int64).sum()) * E > B - len(n) * E
    # Expected fraction for this population is about 0.627.
    assert 0.60 < B / T < 0.66


def test_budget_rule_mixed_entry_sizes():
    n = [100, 200, 300]
    E = [10, 1000, 50]
    B = 100000
    k = oracle.k_budget(n, E, B).tolist()
    T = sum(a * b for a, b in zip(n, E))
    assert k == [a * B // T for a in n]
    assert sum(a * b for a, b in zip(k, E)) <= B


def _golden_kv(name):
    g = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split()
                g[k] = float(v)
    return g


def test_budget_plan_paper_boundary():
    # Sec. 7.5: at 16 MB nothing is evicted; the footprint is 15.4 MB.
    g = _golden_kv("evict_boundary.txt")
    S, n, E = int(g["sessions"]), int(g["frames_per_session"]), int(g["frame_bytes"])
    assert round(S * n * E / 1e6, 1) == g["unconstrained_mb"]
    k, sh, dr = oracle.budget_plan([n] * S, E, int(g["budget_no_evict_mb"] * 1e6), g["keep_fraction"])
    assert (sh, dr) == (0, 0) and k.tolist() == [n] * S
    # Just below the footprint the plan must act, and only as much as needed.
    k, sh, dr = oracle.budget_plan([n] * S, E, S * n * E - 1, g["keep_fraction"])
    assert (sh, dr) == (1, 0) and k.tolist()[0] == 3 and k.tolist()[1:] == [n] * (S - 1)


@pytest.mark.parametrize("seed", range(20))
def test_budget_plan_properties(seed):
    rnd = np.random.default_rng(seed)
    S = int(rnd.integers(1, 40))
    n = rnd.integers(0, 60, S)
    E = rnd.integers(1, 5000, S).astype(np.uint64)
    pr = rnd.permutation(S).astype(np.float64)
    frac = float(rnd.choice([0.0, 0.12, 0.25, 0.5]))
    total = int((n.astype(np.uint64) * E).sum())
    prev = -1
    # Budgets from loose to tight: the plan may only ever do more.
    for B in sorted(set([0, total // 10, total // 3, total // 2, total - 1, total, total + 5]),
                    reverse=True):
        k, sh, dr = oracle.budget_plan(n, E, B, frac, priority=pr)
        kept = int((k.astype(np.uint64) * E).sum())
        target = np.array([min(max(int(np.round(frac * x)), 0), x) for x in n])  # half-even ok: frac*n rarely .5
        assert kept <= B or B >= total
        if B >= total:
            assert (sh, dr) == (0, 0)
        # Drops happen only once every bank that can shrink has been shrunk.
        if dr:
            assert sh == int((target < n).sum())
        # Each bank is whole, at its retention target, or dropped.
        assert all(kk in (nn, tt, 0) for kk, nn, tt in zip(k, n, target))
        # Reactive: acting is monotone in the pressure (tighter budget, more actions).
        assert sh + dr >= prev
        prev = sh + dr


def _global_order(scores):
    # Independent of the oracle: Python's sort on (NaN last, -score, position).
    def rank_key(p):
        s = float(scores[p])
        return (1, 0.0, p) if np.isnan(s) else (0, -s, p)
    return sorted(range(len(scores)), key=rank_key)


def _check_global(scores, n, E, B):
    kept, off = oracle.prune_global(scores, n, E, B)
    starts = np.concatenate([[0], np.cumsum(n)]).astype(np.int64)
    Eb = np.repeat(np.asarray(E, dtype=np.int64), n)
    assert off[0] == 0 and np.all(np.diff(off) >= 0) and off[-1] == kept.size
    chosen = set()
    for b in range(len(n)):
        part = kept[off[b]:off[b + 1]]
        assert np.all(np.diff(part) > 0) and np.all(part >= 0) and np.all(part < n[b])
        chosen.update((starts[b] + part).tolist())
    total = int(Eb.sum())
    used = int(sum(Eb[p] for p in chosen))
    # The kept set is exactly a prefix of the global order ...
    order = _global_order(scores)
    m = len(chosen)
    assert set(order[:m]) == chosen
    # ... within the budget, and the next entry of the order does not fit.
    assert used <= B
    if m < len(order):
        assert used + int(Eb[order[m]]) > B
    else:
        assert total <= B
    return kept, off


@pytest.mark.parametrize("seed", range(40))
def test_prune_global_is_the_longest_fitting_prefix(seed):
    rnd = np.random.default_rng(seed)
    nb = int(rnd.integers(1, 7))
    n = rnd.integers(0, 9, nb).astype(np.int32)
    E = rnd.integers(0, 40, nb).astype(np.uint64)
    pool = np.array([0.5, -0.25, 0.0, -0.0, 1.0, np.nan, 0.5, 0.125], dtype=np.float32)
    s = pool[rnd.integers(0, pool.size, int(n.sum()))]
    total = int((n.astype(np.int64) * E.astype(np.int64)).sum())
    for B in sorted({0, 1, total // 3, total // 2, max(total - 1, 0), total, total + 7}):
        _check_global(s, n, E, B)


def test_prune_global_special_cases():
    rnd = np.random.default_rng(5)
    s = rnd.standard_normal(50).astype(np.float32)
    # One bank, uniform entry bytes: a global threshold is the bank's top-k.
    for k in (0, 1, 7, 49, 50):
        kept, off = oracle.prune_global(s, [50], [3072], k * 3072 + 100)
        assert kept.tolist() == oracle.topk(s, k).tolist()
    # Budget that does not bind keeps everything; zero budget keeps nothing.
    kept, off = oracle.prune_global(s, [20, 0, 30], [8, 8, 8], 50 * 8)
    assert off.tolist() == [0, 20, 20, 50] and kept.tolist() == list(range(20)) + list(range(30))
    kept, off = oracle.prune_global(s, [20, 0, 30], [8, 8, 8], 0)
    assert kept.size == 0 and off.tolist() == [0, 0, 0, 0]
    # Equal scores everywhere: ties go to the lower bank, then the lower index.
    eq = np.full(12, 0.25, dtype=np.float32)
    kept, off = oracle.prune_global(eq, [4, 4, 4], [1, 1, 1], 6)
    assert off.tolist() == [0, 4, 6, 6] and kept.tolist() == [0, 1, 2, 3, 0, 1]
    # A bank of more relevant entries keeps more than the same-fraction rule gives it.
    hi = np.linspace(0.9, 0.8, 10).astype(np.float32)
    lo = np.linspace(0.1, 0.0, 10).astype(np.float32)
    kept, off = oracle.prune_global(np.concatenate([lo, hi]), [10, 10], [5, 5], 50)
    assert off.tolist() == [0, 0, 10]
    assert oracle.k_budget([10, 10], 5, 50).tolist() == [5, 5]
